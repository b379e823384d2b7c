"""AQ-SGD with quantisation (§2.5; the change of each sample's activation against its
buffer, quantised as in §2.2) on the GPU through the C ABI, against the CPU oracle bit for
bit over several steps: codes, scale, min, the sender's buffer and the receiver's copy.
Widths 2/4/6/8 (the paper's) plus the fp32 passthrough, both roundings, rows on the warp,
cluster and two-pass quantiser paths, ragged lengths."""

import numpy as np
import pytest
import torch

import oracle
from gpu_cases import assert_bits_equal

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def mpc():
    import __graft_entry__ as g

    g.build()
    import paper_2401_07788_gb300 as m

    torch.cuda.set_device(0)
    return m


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def run_steps(mpc, S, rps, L, n, bits, stochastic, steps, seed):
    rng = np.random.default_rng(seed)
    buf = np.zeros((S, rps, L), np.float32)
    buf_dev = dev(buf)
    recv_dev = dev(buf)
    base = rng.standard_normal((S, rps, L)).astype(np.float32)
    for step in range(steps):
        ids = rng.permutation(S)[:n].astype(np.int64)
        # the activation of a sample drifts slowly between its visits (§2.5's premise)
        x = (base[ids] + 0.05 * (step + 1) * rng.standard_normal((n, rps, L))).astype(np.float32)
        ids_dev = dev(ids)
        sd = seed * 1000 + step
        c, s, m = mpc.mpc_aqsgd_quant_compress(dev(x), buf_dev, ids_dev, bits,
                                               stochastic=stochastic, seed=sd)
        mpc.mpc_aqsgd_quant_decompress(c, s, m, recv_dev, ids_dev, bits)
        assert mpc.mpc_get_status() == 0, mpc.mpc_last_error()
        oc, os_, om = oracle.aqsgd_quant_compress(x, buf, ids, bits, stochastic, sd)
        what = "bits=%d sr=%d L=%d step %d" % (bits, stochastic, L, step)
        assert_bits_equal(c.cpu().numpy().view(np.uint32), oc, "codes " + what)
        assert_bits_equal(s.cpu().numpy(), os_, "scale " + what)
        assert_bits_equal(m.cpu().numpy(), om, "min " + what)
        assert_bits_equal(buf_dev.cpu().numpy(), buf, "buffer " + what)
        assert_bits_equal(recv_dev.cpu().numpy(), buf, "receiver " + what)


@pytest.mark.parametrize("bits", [2, 4, 6, 8, 32])
@pytest.mark.parametrize("stochastic", [False, True])
def test_aqsgd_quant_widths(mpc, bits, stochastic):
    run_steps(mpc, S=24, rps=2, L=4096, n=6, bits=bits, stochastic=stochastic, steps=3,
              seed=bits * 2 + stochastic)


@pytest.mark.parametrize("L", [1, 7, 1001, 16384, 70001])
def test_aqsgd_quant_lengths(mpc, L):
    run_steps(mpc, S=9, rps=3, L=L, n=4, bits=4, stochastic=True, steps=2, seed=L % 977)


@pytest.mark.parametrize("L", [1, 7, 128, 256, 300, 768, 1024, 1025, 2048, 2049, 3000, 4095, 4096])
@pytest.mark.parametrize("bits,stochastic", [(2, False), (8, True), (4, False)])
def test_aqsgd_quant_one_pass_shapes(mpc, L, bits, stochastic):
    """The one-pass sender (2/4/8-bit codes, rows of up to 4096 entries: a warp per row,
    four warps from 1025 on), ragged lengths included, against the oracle."""
    run_steps(mpc, S=11, rps=3, L=L, n=5, bits=bits, stochastic=stochastic, steps=2,
              seed=L + bits)


def test_aqsgd_quant_cnn_boundary_shape(mpc):
    """The CNN stage boundary: 128 samples of [128, 16, 16] activations, one row per sample,
    drawn from a 512-sample set."""
    run_steps(mpc, S=512, rps=1, L=128 * 16 * 16, n=128, bits=8, stochastic=False, steps=2,
              seed=11)


def test_aqsgd_quant_empty_and_bad_id(mpc):
    S, rps, L = 4, 2, 256
    buf = torch.zeros((S, rps, L), dtype=torch.float32, device="cuda")
    x = torch.ones((0, rps, L), dtype=torch.float32, device="cuda")
    ids = torch.zeros(0, dtype=torch.int64, device="cuda")
    c, s, m = mpc.mpc_aqsgd_quant_compress(x, buf, ids, 4)
    assert c.shape[0] == 0 and mpc.mpc_get_status() == 0
    x = torch.ones((2, rps, L), dtype=torch.float32, device="cuda")
    ids = torch.tensor([1, 9], dtype=torch.int64, device="cuda")
    mpc.mpc_aqsgd_quant_compress(x, buf, ids, 4)
    assert mpc.mpc_get_status() == 6  # MPC_ERR_DEVICE
    assert mpc.mpc_get_status() == 0  # cleared
    # the valid id's rows took the update; no other buffer row was written
    assert bool((buf[1] == 1.0).all()) and float(buf[[0, 2, 3]].abs().sum()) == 0
