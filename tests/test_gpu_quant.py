"""Min-max quantisation on the GPU (through the C ABI) against the CPU oracle, bit for bit:
codes, scale, min and the dequantised rows."""

import numpy as np
import pytest
import torch

import oracle
from gpu_cases import assert_bits_equal, rows_of

pytestmark = pytest.mark.gpu

LENGTHS = [1, 2, 3, 31, 32, 33, 63, 64, 65, 767, 768, 1024, 2047, 2048, 2049, 4097, 8192,
           8193, 16384, 32768, 65535, 65536, 65537, 200003]


@pytest.fixture(scope="module")
def mpc():
    import __graft_entry__ as g

    g.build()
    import paper_2401_07788_gb300 as m

    torch.cuda.set_device(0)
    return m


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def run_both(mpc, x, bits, stochastic, seed):
    R, L = x.shape
    c, s, m = mpc.mpc_quant_compress(dev(x), bits, stochastic=stochastic, seed=seed)
    y = mpc.mpc_quant_decompress(c, s, m, L, bits)
    assert mpc.mpc_get_status() == 0, mpc.mpc_last_error()
    oc, os_, om = oracle.quant_compress(x, bits, stochastic, seed)
    oy = oracle.quant_decompress(oc, os_, om, L, bits)
    tag = "bits=%d L=%d sr=%s" % (bits, L, stochastic)
    assert_bits_equal(c.cpu().numpy().view(np.uint32), oc, "codes " + tag)
    assert_bits_equal(s.cpu().numpy(), os_, "scale " + tag)
    assert_bits_equal(m.cpu().numpy(), om, "minv " + tag)
    assert_bits_equal(y.cpu().numpy(), oy, "dequant " + tag)


@pytest.mark.parametrize("L", LENGTHS)
@pytest.mark.parametrize("bits", [2, 4, 8, 32])
def test_quant_lengths(mpc, L, bits):
    x = rows_of("normal", 3, L, seed=L)
    for stochastic in (False, True):
        run_both(mpc, x, bits, stochastic, seed=(5 << 32) | 17)


@pytest.mark.parametrize("kind", ["relu", "zeros", "equal", "ties", "signed_zero", "heavy",
                                  "outlier"])
@pytest.mark.parametrize("bits", [2, 4, 8])
def test_quant_kinds(mpc, kind, bits):
    for L in (768, 5000, 32768):
        x = rows_of(kind, 4, L, seed=3)
        for stochastic in (False, True):
            run_both(mpc, x, bits, stochastic, seed=123)


@pytest.mark.parametrize("R,L", [(500, 768), (64, 4096), (130, 32768), (7, 1001)])
def test_quant_many_rows(mpc, R, L):
    x = (rows_of("normal", R, L, seed=R) * 1e-3).astype(np.float32)
    for bits in (2, 4, 8):
        run_both(mpc, x, bits, True, seed=(3 << 32) | 9)
        run_both(mpc, x, bits, False, seed=0)


def test_quant_seed_changes_codes(mpc):
    x = dev(rows_of("normal", 2, 4096, seed=1))
    a = mpc.mpc_quant_compress(x, 4, stochastic=True, seed=1)[0]
    b = mpc.mpc_quant_compress(x, 4, stochastic=True, seed=1)[0]
    c = mpc.mpc_quant_compress(x, 4, stochastic=True, seed=2)[0]
    assert torch.equal(a, b) and not torch.equal(a, c)


# Rows of 8193..32768 entries with enough rows to fill the GPU in one wave take one wide
# CTA each (512 threads up to 16384 entries, else 1024): every width, both roundings,
# aligned and unaligned rows, degenerate rows.
@pytest.mark.parametrize("R,L", [(160, 8193), (160, 16384), (200, 12345), (120, 16385),
                                 (116, 20001), (128, 32768)])
def test_quant_wide_rows(mpc, R, L):
    for kind in ("normal", "relu", "equal"):
        x = rows_of(kind, R, L, seed=L)
        for bits in (1, 2, 4, 6, 8, 13, 16, 32):
            run_both(mpc, x, bits, False, seed=0)
        for bits in (2, 6, 8):
            run_both(mpc, x, bits, True, seed=(7 << 32) | L)
