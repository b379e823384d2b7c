"""TopK, error feedback, EF21 and AQ-SGD on the GPU (through the C ABI) against the CPU
oracle, bit for bit: indices, values, error and state buffers, decompressed rows."""

import numpy as np
import pytest
import torch

import oracle
from gpu_cases import KINDS, assert_bits_equal, rows_of

pytestmark = pytest.mark.gpu

LENGTHS = [1, 5, 31, 32, 33, 127, 128, 129, 767, 768, 769, 1024, 2047, 2048, 2049, 4095,
           4096, 4097, 8191, 8192, 8193, 16384, 32768, 65535, 65536]


@pytest.fixture(scope="module")
def mpc():
    import __graft_entry__ as g

    g.build()
    import paper_2401_07788_gb300 as m

    torch.cuda.set_device(0)
    return m


def ks_for(L):
    return sorted({1, max(1, L // 10), max(1, L - 1), L})


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def check_status(mpc):
    st = mpc.mpc_get_status()
    assert st == 0, mpc.mpc_last_error()


@pytest.mark.parametrize("L", LENGTHS)
def test_topk_lengths(mpc, L):
    R = 3
    for kind in ("normal", "relu", "ties"):
        x = rows_of(kind, R, L, seed=L)
        xd = dev(x)
        for k in ks_for(L):
            v, i = mpc.mpc_topk_compress(xd, k)
            y = mpc.mpc_topk_decompress(v, i, L)
            check_status(mpc)
            ov, oi = oracle.topk_compress(x, k)
            assert_bits_equal(i.cpu().numpy(), oi, "idx L=%d k=%d %s" % (L, k, kind))
            assert_bits_equal(v.cpu().numpy(), ov, "vals L=%d k=%d %s" % (L, k, kind))
            assert_bits_equal(y.cpu().numpy(), oracle.topk_decompress(ov, oi, L),
                              "decompress L=%d k=%d %s" % (L, k, kind))


@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("L", [768, 1000, 4096, 16384, 65536])
def test_topk_value_kinds(mpc, kind, L):
    R = 4
    x = rows_of(kind, R, L, seed=7)
    xd = dev(x)
    for k in (1, max(1, L // 100), max(1, L // 10), L // 2, L - 1):
        v, i = mpc.mpc_topk_compress(xd, k)
        check_status(mpc)
        ov, oi = oracle.topk_compress(x, k)
        assert_bits_equal(i.cpu().numpy(), oi, "idx %s L=%d k=%d" % (kind, L, k))
        assert_bits_equal(v.cpu().numpy(), ov, "vals %s L=%d k=%d" % (kind, L, k))


@pytest.mark.parametrize("R,L,pct", [(200, 768, 10), (300, 1024, 30), (64, 4096, 1),
                                     (40, 16384, 10), (9, 32768, 5), (3, 65536, 50),
                                     (1000, 33, 10), (2, 12345, 10)])
def test_topk_many_rows(mpc, R, L, pct):
    x = rows_of("normal", R, L, seed=R + L)
    k = max(1, L * pct // 100)
    v, i = mpc.mpc_topk_compress(dev(x), k)
    check_status(mpc)
    ov, oi = oracle.topk_compress(x, k)
    assert_bits_equal(i.cpu().numpy(), oi, "idx")
    assert_bits_equal(v.cpu().numpy(), ov, "vals")


@pytest.mark.parametrize("L,R", [(768, 33), (1000, 5), (4096, 6), (16384, 4), (32768, 3),
                                 (65536, 2), (129, 17)])
def test_ef_multistep(mpc, L, R):
    rng = np.random.default_rng(L)
    k = max(1, L // 10)
    e_host = np.zeros((R, L), np.float32)
    e_dev = torch.zeros((R, L), dtype=torch.float32, device="cuda")
    x = np.maximum(rng.standard_normal((R, L)), 0).astype(np.float32)
    for step in range(4):
        v, i = mpc.mpc_ef_topk_compress(dev(x), e_dev, k)
        check_status(mpc)
        ov, oi = oracle.ef_topk_compress(x, e_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "EF vals step %d" % step)
        assert_bits_equal(e_dev.cpu().numpy(), e_host, "EF err step %d" % step)
        x = (x + 0.1 * rng.standard_normal((R, L))).astype(np.float32)


@pytest.mark.parametrize("L,R", [(768, 40), (1024, 9), (999, 7), (4096, 5), (16384, 3),
                                 (65536, 2)])
def test_ef21_multistep(mpc, L, R):
    rng = np.random.default_rng(L + 1)
    k = max(1, L // 10)
    g_host = np.zeros((R, L), np.float32)
    g_dev = torch.zeros((R, L), dtype=torch.float32, device="cuda")
    x = rng.standard_normal((R, L)).astype(np.float32)
    for step in range(4):
        v, i = mpc.mpc_ef21_topk_compress(dev(x), g_dev, k)
        check_status(mpc)
        ov, oi = oracle.ef21_topk_compress(x, g_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF21 idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "EF21 vals step %d" % step)
        assert_bits_equal(g_dev.cpu().numpy(), g_host, "EF21 g step %d" % step)
        x = (x + 0.05 * rng.standard_normal((R, L))).astype(np.float32)


@pytest.mark.parametrize("L", [1024, 768, 1001, 4096, 20000])
def test_aqsgd(mpc, L):
    rng = np.random.default_rng(L + 2)
    S, rps, n = 40, 3, 7
    k = max(1, L * 30 // 100)
    buf = rng.standard_normal((S, rps, L)).astype(np.float32)
    buf_dev = dev(buf)
    recv_dev = dev(buf)
    for step in range(3):
        ids = rng.permutation(S)[:n].astype(np.int64)
        x = (buf[ids] + 0.05 * rng.standard_normal((n, rps, L))).astype(np.float32)
        ids_dev = dev(ids)
        v, i = mpc.mpc_aqsgd_compress(dev(x), buf_dev, ids_dev, k)
        mpc.mpc_aqsgd_decompress(v, i, recv_dev, ids_dev)
        check_status(mpc)
        ov, oi = oracle.aqsgd_compress(x, buf, ids, k)
        assert_bits_equal(i.cpu().numpy(), oi, "AQ-SGD idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "AQ-SGD vals step %d" % step)
        assert_bits_equal(buf_dev.cpu().numpy(), buf, "AQ-SGD buffer step %d" % step)
        assert_bits_equal(recv_dev.cpu().numpy(), buf, "AQ-SGD receiver step %d" % step)


def test_aqsgd_bad_id_reports(mpc):
    S, rps, L, k = 4, 2, 256, 20
    buf = torch.zeros((S, rps, L), dtype=torch.float32, device="cuda")
    x = torch.ones((2, rps, L), dtype=torch.float32, device="cuda")
    ids = torch.tensor([1, 9], dtype=torch.int64, device="cuda")
    mpc.mpc_aqsgd_compress(x, buf, ids, k)
    assert mpc.mpc_get_status() == 6  # MPC_ERR_DEVICE
    assert mpc.mpc_get_status() == 0  # cleared
    # the valid id's rows were processed
    assert float(buf[1].abs().sum()) > 0 and float(buf[[0, 2, 3]].abs().sum()) == 0


def test_decompress_garbage_indices_stay_in_bounds(mpc):
    R, L, k = 3, 5000, 40
    vals = torch.ones((R, k), dtype=torch.float32, device="cuda")
    idx = torch.randint(-10**6, 10**6, (R, k), dtype=torch.int32, device="cuda")
    guard = torch.full((R * L + 4096,), 7.0, device="cuda")
    y = guard[: R * L].view(R, L)
    mpc.mpc_topk_decompress(vals, idx, L, y=y)
    torch.cuda.synchronize()
    assert bool((guard[R * L:] == 7.0).all())


def test_long_row_decompress_tiles(mpc):
    """Rows longer than one output tile: the kept entries of each tile are found by the
    block-parallel search."""
    R, L = 2, 100003
    rng = np.random.default_rng(5)
    for k in (1, 7, 5000, L):
        idx = np.stack([np.sort(rng.choice(L, k, replace=False)) for _ in range(R)]).astype(np.int32)
        vals = rng.standard_normal((R, k)).astype(np.float32)
        y = mpc.mpc_topk_decompress(dev(vals), dev(idx), L)
        assert_bits_equal(y.cpu().numpy(), oracle.topk_decompress(vals, idx, L), "k=%d" % k)


@pytest.mark.parametrize("R,L", [(4096, 768), (3000, 8192), (5, 8193), (3, 3000001),
                                 (2, 1 << 22)])
def test_decompress_tiles_cross_rows(mpc, R, L):
    """Output tiles of whole short rows (the row of a payload entry found by a high
    product), rows of exactly one tile, and long rows split into more tiles than there are
    CTAs, so that a CTA starts inside a row and carries on across row boundaries."""
    rng = np.random.default_rng(L)
    for k in sorted({1, 3, L // 100 + 1, L // 2, L}):
        idx = np.sort(np.stack([rng.choice(L, k, replace=False) for _ in range(R)]),
                      axis=1).astype(np.int32) if k < L else np.tile(np.arange(L, dtype=np.int32), (R, 1))
        vals = rng.standard_normal((R, k)).astype(np.float32)
        y = mpc.mpc_topk_decompress(dev(vals), dev(idx), L)
        assert_bits_equal(y.cpu().numpy(), oracle.topk_decompress(vals, idx, L),
                          "R=%d L=%d k=%d" % (R, L, k))


# Rows of 8193..32768 entries with enough rows to fill the GPU take one wide CTA each
# (512 threads up to 16384 entries, else 1024); the knob value 3 keeps them on clusters.
WIDE = [(160, 8192), (160, 8193), (160, 12345), (160, 16384), (120, 16385), (116, 20000),
        (120, 32768), (300, 9000)]


@pytest.mark.parametrize("R,L", WIDE)
@pytest.mark.parametrize("path", [0, 3])
def test_topk_wide_rows(mpc, R, L, path):
    try:
        mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, path)
        for kind in ("normal", "relu", "ties", "zeros", "outlier"):
            x = rows_of(kind, R, L, seed=L + R)
            xd = dev(x)
            for k in (1, L // 20, L // 3, L - 1):
                v, i = mpc.mpc_topk_compress(xd, k)
                check_status(mpc)
                ov, oi = oracle.topk_compress(x, k)
                assert_bits_equal(i.cpu().numpy(), oi, "idx %s L=%d k=%d" % (kind, L, k))
                assert_bits_equal(v.cpu().numpy(), ov, "vals %s L=%d k=%d" % (kind, L, k))
    finally:
        mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, 0)


@pytest.mark.parametrize("R,L", [(160, 16384), (120, 32768), (116, 24001)])
def test_ef_ef21_wide_rows(mpc, R, L):
    rng = np.random.default_rng(L)
    k = max(1, L // 10)
    e_host = np.zeros((R, L), np.float32)
    g_host = np.zeros((R, L), np.float32)
    e_dev = torch.zeros((R, L), dtype=torch.float32, device="cuda")
    g_dev = torch.zeros((R, L), dtype=torch.float32, device="cuda")
    x = np.maximum(rng.standard_normal((R, L)), 0).astype(np.float32)
    for step in range(3):
        v, i = mpc.mpc_ef_topk_compress(dev(x), e_dev, k)
        check_status(mpc)
        ov, oi = oracle.ef_topk_compress(x, e_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "EF vals step %d" % step)
        assert_bits_equal(e_dev.cpu().numpy(), e_host, "EF err step %d" % step)
        v, i = mpc.mpc_ef21_topk_compress(dev(x), g_dev, k)
        check_status(mpc)
        ov, oi = oracle.ef21_topk_compress(x, g_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF21 idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "EF21 vals step %d" % step)
        assert_bits_equal(g_dev.cpu().numpy(), g_host, "EF21 g step %d" % step)
        x = (x + 0.1 * rng.standard_normal((R, L))).astype(np.float32)


def test_aqsgd_wide_rows(mpc):
    """AQ-SGD rows of 16384 entries, 160 of them (8 samples x 20 rows): one wide CTA a row."""
    rng = np.random.default_rng(3)
    S, rps, n, L = 24, 20, 8, 16384
    k = L * 30 // 100
    buf = rng.standard_normal((S, rps, L)).astype(np.float32)
    buf_dev = dev(buf)
    for step in range(2):
        ids = rng.permutation(S)[:n].astype(np.int64)
        x = (buf[ids] + 0.05 * rng.standard_normal((n, rps, L))).astype(np.float32)
        v, i = mpc.mpc_aqsgd_compress(dev(x), buf_dev, dev(ids), k)
        check_status(mpc)
        ov, oi = oracle.aqsgd_compress(x, buf, ids, k)
        assert_bits_equal(i.cpu().numpy(), oi, "AQ-SGD idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "AQ-SGD vals step %d" % step)
        assert_bits_equal(buf_dev.cpu().numpy(), buf, "AQ-SGD buffer step %d" % step)
