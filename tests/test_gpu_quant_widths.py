"""Min-max quantisation at every code width 1..16 (§2.2 evaluates 6-bit gradients; widths
that do not divide 32 have codes straddling two words) on the GPU through the C ABI,
against the CPU oracle bit for bit: codes, scale, min and the dequantised rows, on the
warp, cluster and two-pass paths, aligned and unaligned."""

import numpy as np
import pytest
import torch

import oracle
from gpu_cases import assert_bits_equal, rows_of

pytestmark = pytest.mark.gpu

WIDTHS = [1, 3, 5, 6, 7, 9, 10, 11, 12, 13, 15, 16]


@pytest.fixture(scope="module")
def mpc():
    import __graft_entry__ as g

    g.build()
    import paper_2401_07788_gb300 as m

    torch.cuda.set_device(0)
    return m


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def run_both(mpc, x, bits, stochastic, seed, xdev=None):
    R, L = x.shape
    c, s, m = mpc.mpc_quant_compress(dev(x) if xdev is None else xdev, bits,
                                     stochastic=stochastic, seed=seed)
    y = mpc.mpc_quant_decompress(c, s, m, L, bits)
    assert mpc.mpc_get_status() == 0, mpc.mpc_last_error()
    oc, os_, om = oracle.quant_compress(x, bits, stochastic, seed)
    oy = oracle.quant_decompress(oc, os_, om, L, bits)
    tag = "bits=%d L=%d sr=%s" % (bits, L, stochastic)
    assert_bits_equal(c.cpu().numpy().view(np.uint32), oc, "codes " + tag)
    assert_bits_equal(s.cpu().numpy(), os_, "scale " + tag)
    assert_bits_equal(m.cpu().numpy(), om, "minv " + tag)
    assert_bits_equal(y.cpu().numpy(), oy, "dequant " + tag)
    return c, s, m


@pytest.mark.parametrize("bits", WIDTHS)
@pytest.mark.parametrize("L", [1, 5, 31, 33, 128, 767, 2048, 2049, 8192, 32768, 65537])
def test_widths_lengths(mpc, bits, L):
    x = rows_of("normal", 3, L, seed=L + bits)
    for stochastic in (False, True):
        run_both(mpc, x, bits, stochastic, seed=(7 << 32) | bits)


@pytest.mark.parametrize("bits", [6, 12])
@pytest.mark.parametrize("kind", ["relu", "zeros", "equal", "signed_zero", "heavy", "outlier"])
def test_widths_kinds(mpc, bits, kind):
    for L in (768, 5000):
        x = rows_of(kind, 4, L, seed=5)
        for stochastic in (False, True):
            run_both(mpc, x, bits, stochastic, seed=99)


@pytest.mark.parametrize("bits", [3, 6, 16])
def test_widths_unaligned_dequant(mpc, bits):
    """Output rows that are not 16-byte aligned take the one-entry-per-thread path."""
    R, L = 5, 1003
    x = rows_of("normal", R, L, seed=bits)
    c, s, m = run_both(mpc, x, bits, False, seed=0)
    y = torch.zeros(R * L + 1, device="cuda")[1:].view(R, L)
    mpc.mpc_quant_decompress(c, s, m, L, bits, y=y)
    assert mpc.mpc_get_status() == 0, mpc.mpc_last_error()
    oc, os_, om = oracle.quant_compress(x, bits, False, 0)
    assert_bits_equal(y.cpu().numpy(), oracle.quant_decompress(oc, os_, om, L, bits), "unaligned")


def test_six_bit_transformer_boundary_rows(mpc):
    """fw4-bw6 (Table 1): 6-bit gradients of the transformer boundary, per-token rows."""
    from paper_2401_07788_gb300 import synth

    g = synth.normal((8192, 768), 7, "cuda", std=1e-4)
    c, s, m = mpc.mpc_quant_compress(g, 6, stochastic=False)
    y = mpc.mpc_quant_decompress(c, s, m, 768, 6)
    assert mpc.mpc_get_status() == 0, mpc.mpc_last_error()
    rows = np.random.default_rng(0).choice(8192, 64, replace=False)
    gn = g.cpu().numpy()[rows]
    oc, os_, om = oracle.quant_compress(gn, 6)
    W = oracle.quant_row_words(768, 6)
    assert_bits_equal(c.cpu().numpy().view(np.uint32).reshape(8192, W)[rows], oc, "codes")
    assert_bits_equal(y.cpu().numpy()[rows], oracle.quant_decompress(oc, os_, om, 768, 6), "y")
