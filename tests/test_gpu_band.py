"""The band kernel for rows of 1025..8192 entries (the default there) and the cluster /
CTA kernels it replaces (MPC_KNOB_TOPK_PATH = 4), each against the CPU oracle, bit for
bit: edge lengths, value kinds that defeat the sampled band (ties, zeros, equal values, a
far outlier, heavy tails) and so take the exact fallback, every fused variant over
several steps of state, and AQ-SGD's sample-id map."""

import numpy as np
import pytest
import torch

import oracle
from gpu_cases import KINDS, assert_bits_equal, rows_of

pytestmark = pytest.mark.gpu

LENGTHS = [1025, 1027, 1028, 1536, 2047, 2048, 2049, 3000, 4095, 4096, 4097, 5000, 8188,
           8191, 8192]


@pytest.fixture(scope="module")
def mpc():
    import __graft_entry__ as g

    g.build()
    import paper_2401_07788_gb300 as m

    torch.cuda.set_device(0)
    yield m
    m.mpc_set_knob(m.MPC_KNOB_TOPK_PATH, 0)


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def ok(mpc):
    assert mpc.mpc_get_status() == 0, mpc.mpc_last_error()


@pytest.mark.parametrize("path", [0, 4])
@pytest.mark.parametrize("L", LENGTHS)
def test_lengths(mpc, L, path):
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, path)
    R = 37
    for kind in ("normal", "relu"):
        x = rows_of(kind, R, L, seed=L + 3)
        xd = dev(x)
        for k in sorted({1, L // 100 or 1, L // 10, L // 3, L // 2, L // 2 + 1, (3 * L) // 4,
                         L - 1, L}):
            v, i = mpc.mpc_topk_compress(xd, k)
            ok(mpc)
            ov, oi = oracle.topk_compress(x, k)
            assert_bits_equal(i.cpu().numpy(), oi, "idx %s L=%d k=%d" % (kind, L, k))
            assert_bits_equal(v.cpu().numpy(), ov, "vals %s L=%d k=%d" % (kind, L, k))


@pytest.mark.parametrize("path", [0, 4])
@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("L", [1100, 4096, 8192])
def test_value_kinds(mpc, kind, L, path):
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, path)
    R = 9
    x = rows_of(kind, R, L, seed=11)
    xd = dev(x)
    for k in (1, L // 100, L // 10, L // 2, L - 1):
        k = max(1, k)
        v, i = mpc.mpc_topk_compress(xd, k)
        ok(mpc)
        ov, oi = oracle.topk_compress(x, k)
        assert_bits_equal(i.cpu().numpy(), oi, "idx %s L=%d k=%d" % (kind, L, k))
        assert_bits_equal(v.cpu().numpy(), ov, "vals %s L=%d k=%d" % (kind, L, k))


@pytest.mark.parametrize("path", [0, 4])
@pytest.mark.parametrize("L,R,pct", [(4096, 300, 1), (4096, 300, 10), (4096, 300, 50),
                                     (2048, 200, 10), (8192, 150, 30), (1028, 90, 5),
                                     (6001, 40, 20)])
def test_fused_multistep(mpc, L, R, pct, path):
    """Error feedback and EF21 over four drifting steps (state carried on both sides)."""
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, path)
    rng = np.random.default_rng(L + R + pct)
    k = max(1, L * pct // 100)
    e_host = np.zeros((R, L), np.float32)
    g_host = np.zeros((R, L), np.float32)
    e_dev = torch.zeros((R, L), device="cuda")
    g_dev = torch.zeros((R, L), device="cuda")
    x = rng.standard_normal((R, L)).astype(np.float32)
    for step in range(4):
        xd = dev(x)
        v, i = mpc.mpc_ef_topk_compress(xd, e_dev, k)
        ok(mpc)
        ov, oi = oracle.ef_topk_compress(x, e_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "EF vals step %d" % step)
        assert_bits_equal(e_dev.cpu().numpy(), e_host, "EF err step %d" % step)
        v, i = mpc.mpc_ef21_topk_compress(xd, g_dev, k)
        ok(mpc)
        ov, oi = oracle.ef21_topk_compress(x, g_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF21 idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "EF21 vals step %d" % step)
        assert_bits_equal(g_dev.cpu().numpy(), g_host, "EF21 g step %d" % step)
        x = (x + 0.1 * rng.standard_normal((R, L))).astype(np.float32)


@pytest.mark.parametrize("path", [0, 4])
def test_aqsgd_ids(mpc, path):
    """AQ-SGD rows of 4096 entries through the sample-id map, and an unaligned row length."""
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, path)
    rng = np.random.default_rng(5)
    for L in (4096, 4097):
        S, rps, n = 12, 7, 5
        k = L * 30 // 100
        buf = rng.standard_normal((S, rps, L)).astype(np.float32)
        buf_dev = dev(buf)
        for step in range(2):
            ids = rng.permutation(S)[:n].astype(np.int64)
            x = (buf[ids] + 0.05 * rng.standard_normal((n, rps, L))).astype(np.float32)
            v, i = mpc.mpc_aqsgd_compress(dev(x), buf_dev, dev(ids), k)
            ok(mpc)
            ov, oi = oracle.aqsgd_compress(x, buf, ids, k)
            assert_bits_equal(i.cpu().numpy(), oi, "idx L=%d step %d" % (L, step))
            assert_bits_equal(v.cpu().numpy(), ov, "vals L=%d step %d" % (L, step))
            assert_bits_equal(buf_dev.cpu().numpy(), buf, "buffer L=%d step %d" % (L, step))


@pytest.mark.parametrize("path", [0, 4])
def test_unaligned_pointer(mpc, path):
    """A row base that is 4- but not 16-byte aligned takes plain loads."""
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, path)
    R, L = 21, 4096
    x = rows_of("normal", R, L + 1, seed=3)[:, 1:]
    flat = torch.from_numpy(np.ascontiguousarray(rows_of("normal", 1, R * L + 1, seed=3))).cuda()
    xd = flat[0, 1:].view(R, L)
    xh = xd.cpu().numpy()
    e_dev = torch.zeros((R * L + 1,), device="cuda")[1:].view(R, L)
    e_host = np.zeros((R, L), np.float32)
    for k in (41, 409, 2048):
        v, i = mpc.mpc_topk_compress(xd, k)
        ok(mpc)
        ov, oi = oracle.topk_compress(xh, k)
        assert_bits_equal(i.cpu().numpy(), oi, "idx k=%d" % k)
        assert_bits_equal(v.cpu().numpy(), ov, "vals k=%d" % k)
        v, i = mpc.mpc_ef_topk_compress(xd, e_dev, k)
        ok(mpc)
        ov, oi = oracle.ef_topk_compress(xh, e_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF idx k=%d" % k)
        assert_bits_equal(e_dev.cpu().numpy(), e_host, "EF err k=%d" % k)
    del x
