"""The two-pass row kernel for aligned rows of 8193..65536 entries (the default there)
and the cluster / wide-CTA kernels it replaces (MPC_KNOB_TOPK_PATH = 3), each against the
CPU oracle, bit for bit: edge lengths and k, value kinds that defeat the sampled band
(ties, zeros, equal values, a far outlier, heavy tails, a sample that sees only outliers)
and so take the exact selection over the row, ties at the threshold inside the band,
every fused variant over several steps of state, and AQ-SGD's sample-id map."""

import numpy as np
import pytest
import torch

import oracle
from gpu_cases import KINDS, assert_bits_equal, row_blocks, rows_of

pytestmark = pytest.mark.gpu

LENGTHS = [8196, 8200, 10000, 12288, 16384, 16388, 20000, 32768, 40000, 65532, 65536]


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


def check_topk(mpc, x, k, what):
    v, i = mpc.mpc_topk_compress(dev(x), k)
    ok(mpc)
    ov, oi = row_blocks(lambda b: oracle.topk_compress(b, k), x.shape[0], x)
    assert_bits_equal(i.cpu().numpy(), oi, "idx " + what)
    assert_bits_equal(v.cpu().numpy(), ov, "vals " + what)


@pytest.mark.parametrize("path", [0, 3])
@pytest.mark.parametrize("L", LENGTHS)
def test_lengths(mpc, L, path):
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, path)
    R = 11
    for kind in ("normal", "relu"):
        x = rows_of(kind, R, L, seed=L + 5)
        for k in sorted({1, L // 100, L // 10, L // 3, L // 2, L // 2 + 1, (3 * L) // 4,
                         L - 1, L}):
            check_topk(mpc, x, k, "%s L=%d k=%d" % (kind, L, k))


@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("L", [12288, 65536])
def test_value_kinds(mpc, kind, L):
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, 0)
    x = rows_of(kind, 7, L, seed=13)
    for k in (1, L // 100, L // 10, L // 2, L - 1):
        check_topk(mpc, x, k, "%s L=%d k=%d" % (kind, L, k))


def sample_positions(L):
    """The entries the kernel samples: one float4 group per thread of 512, evenly spread."""
    step = (L // 4 // 512) * 4
    return (np.arange(512)[:, None] * step + np.arange(4)[None, :]).ravel()


@pytest.mark.parametrize("scale", [1000.0, 1e-3])
@pytest.mark.parametrize("L", [16384, 65536])
def test_sample_misled(mpc, L, scale):
    """Outliers (or tiny values) at exactly the sampled entries: the band misses, or the
    one-pass list overflows, and the exact selection over the row runs, for every
    variant."""
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, 0)
    R = 5
    rng = np.random.default_rng(L)
    x = rng.standard_normal((R, L)).astype(np.float32)
    x[:, sample_positions(L)] *= np.float32(scale)
    for k in (L // 100, L // 10, L // 2):
        check_topk(mpc, x, k, "misled L=%d k=%d" % (L, k))
        e_host = rng.standard_normal((R, L)).astype(np.float32) * 0.1
        e_dev = dev(e_host)
        v, i = mpc.mpc_ef_topk_compress(dev(x), e_dev, k)
        ok(mpc)
        ov, oi = oracle.ef_topk_compress(x, e_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF idx misled k=%d" % k)
        assert_bits_equal(v.cpu().numpy(), ov, "EF vals misled k=%d" % k)
        assert_bits_equal(e_dev.cpu().numpy(), e_host, "EF err misled k=%d" % k)
        g_host = rng.standard_normal((R, L)).astype(np.float32) * 0.1
        g_dev = dev(g_host)
        v, i = mpc.mpc_ef21_topk_compress(dev(x), g_dev, k)
        ok(mpc)
        ov, oi = oracle.ef21_topk_compress(x, g_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF21 idx misled k=%d" % k)
        assert_bits_equal(g_dev.cpu().numpy(), g_host, "EF21 g misled k=%d" % k)


@pytest.mark.parametrize("L", [16384, 65536])
def test_ties_in_band(mpc, L):
    """Values rounded to a grid: every magnitude has many copies, so the k-th is tied
    inside the band and the first ties in index order are kept."""
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, 0)
    rng = np.random.default_rng(L + 1)
    for grid in (0.01, 0.001):
        x = (np.round(rng.standard_normal((9, L)) / grid) * grid).astype(np.float32)
        for k in (L // 100 + 7, L // 10 + 3, L // 2 + 1, L // 3):
            check_topk(mpc, x, k, "grid %g L=%d k=%d" % (grid, L, k))


@pytest.mark.parametrize("path", [0, 3])
@pytest.mark.parametrize("L,R,pct", [(65536, 40, 1), (65536, 40, 10), (65536, 40, 50),
                                     (16384, 120, 30), (20000, 30, 5), (32768, 64, 90),
                                     (16384, 20, 100)])
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
        ov, oi = row_blocks(lambda b, e: oracle.ef_topk_compress(b, e, k), R, x, e_host)
        assert_bits_equal(i.cpu().numpy(), oi, "EF idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "EF vals step %d" % step)
        assert_bits_equal(e_dev.cpu().numpy(), e_host, "EF err step %d" % step)
        v, i = mpc.mpc_ef21_topk_compress(xd, g_dev, k)
        ok(mpc)
        ov, oi = row_blocks(lambda b, g: oracle.ef21_topk_compress(b, g, k), R, x, g_host)
        assert_bits_equal(i.cpu().numpy(), oi, "EF21 idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "EF21 vals step %d" % step)
        assert_bits_equal(g_dev.cpu().numpy(), g_host, "EF21 g step %d" % step)
        x = (x + 0.1 * rng.standard_normal((R, L))).astype(np.float32)


@pytest.mark.parametrize("L", [16384, 65536, 16385])
def test_aqsgd_ids(mpc, L):
    """AQ-SGD through the sample-id map (16385: an unaligned row takes the other kernels)."""
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, 0)
    rng = np.random.default_rng(L)
    S, rps, n = 10, 3, 4
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


@pytest.mark.parametrize("base", ["zeros", "normal"])
@pytest.mark.parametrize("L", [16384, 65536])
def test_infinite_marks(mpc, L, base):
    """+inf entries (EF-mixed TopK marks the input's share with them) rank above every
    finite one, on the sampled path and on the exact selection (an all-zero sample)."""
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, 0)
    rng = np.random.default_rng(L + len(base))
    R = 4
    x = rows_of(base, R, L, seed=L)
    for c in (1, 7, L // 50):
        xi = x.copy()
        for r in range(R):
            xi[r, rng.choice(L, c, replace=False)] = np.inf
        for k in sorted({c, c + 10, L // 10}):
            check_topk(mpc, xi, k, "%s inf=%d L=%d k=%d" % (base, c, L, k))
