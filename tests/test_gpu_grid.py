"""The multi-pass TopK path (rows longer than one thread-block cluster holds, whole
tensors) against the CPU oracle, bit for bit; at 2^30 entries, by the properties that fix
the result at any size."""

import numpy as np
import pytest
import torch

import oracle
from gpu_cases import KINDS, assert_bits_equal, rows_of

pytestmark = pytest.mark.gpu


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


@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("L", [1, 33, 5000, 65537, 100003])
def test_forced_grid_path_kinds(mpc, kind, L):
    """Short rows through the multi-pass path (forced): the candidate list, the
    refinement rounds and the tie handling on every value distribution."""
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, 2)
    try:
        R = 2
        x = rows_of(kind, R, L, seed=L + 3)
        for k in sorted({1, max(1, L // 100), max(1, L // 10), max(1, L // 2), L}):
            v, i = mpc.mpc_topk_compress(dev(x), k)
            ok(mpc)
            ov, oi = oracle.topk_compress(x, k)
            assert_bits_equal(i.cpu().numpy(), oi, "idx %s L=%d k=%d" % (kind, L, k))
            assert_bits_equal(v.cpu().numpy(), ov, "vals %s L=%d k=%d" % (kind, L, k))
    finally:
        mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, 0)


@pytest.mark.parametrize("L", [70001, 131072, 1 << 20])
def test_long_rows_ef_and_ef21(mpc, L):
    rng = np.random.default_rng(L)
    R = 2
    k = max(1, L // 10)
    e_host = np.zeros((R, L), np.float32)
    g_host = np.zeros((R, L), np.float32)
    e_dev = torch.zeros((R, L), device="cuda")
    g_dev = torch.zeros((R, L), device="cuda")
    x = rng.standard_normal((R, L)).astype(np.float32)
    for step in range(2):
        v, i = mpc.mpc_ef_topk_compress(dev(x), e_dev, k)
        ok(mpc)
        ov, oi = oracle.ef_topk_compress(x, e_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF idx")
        assert_bits_equal(v.cpu().numpy(), ov, "EF vals")
        assert_bits_equal(e_dev.cpu().numpy(), e_host, "EF err")
        v, i = mpc.mpc_ef21_topk_compress(dev(x), g_dev, k)
        ok(mpc)
        ov, oi = oracle.ef21_topk_compress(x, g_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF21 idx")
        assert_bits_equal(g_dev.cpu().numpy(), g_host, "EF21 g")
        x = (x + 0.1 * rng.standard_normal((R, L))).astype(np.float32)


@pytest.mark.parametrize("pct", [1, 10, 50])
def test_whole_tensor_2p24(mpc, pct):
    """One row of 2^24 entries (a whole 64 MiB tensor), plain TopK, against the oracle."""
    from paper_2401_07788_gb300 import synth

    N = 1 << 24
    x = synth.normal((1, N), 24, "cuda")
    k = synth.k_of(N, pct)
    v, i = mpc.mpc_topk_compress(x, k)
    y = mpc.mpc_topk_decompress(v, i, N)
    ok(mpc)
    xn = x.cpu().numpy()
    ov, oi = oracle.topk_compress(xn, k)
    assert_bits_equal(i.cpu().numpy(), oi, "idx")
    assert_bits_equal(v.cpu().numpy(), ov, "vals")
    assert_bits_equal(y.cpu().numpy(), oracle.topk_decompress(ov, oi, N), "decompress")


@pytest.mark.parametrize("pct", [1, 50])
def test_whole_tensor_2p30_properties(mpc, pct):
    """One row of 2^30 entries: exactly k entries, strictly ascending indices, values
    equal to x at those indices, every kept magnitude >= every dropped one, and among
    entries at the threshold magnitude the lowest indices are the kept ones."""
    from paper_2401_07788_gb300 import synth

    N = 1 << 30
    x = synth.normal((1, N), 30, "cuda")
    x[0, 12345:12345 + 1000] = 0.5  # a block of equal magnitudes
    k = synth.k_of(N, pct)
    v, i = mpc.mpc_topk_compress(x, k)
    ok(mpc)
    i64 = i[0].long()
    assert i64.numel() == k
    assert bool((i64[1:] > i64[:-1]).all())
    assert bool((i64[0] >= 0) & (i64[-1] < N))
    assert torch.equal(v[0].view(torch.int32), x[0, i64].view(torch.int32))
    kept = torch.zeros(N, dtype=torch.bool, device="cuda")
    kept[i64] = True
    a = x[0].abs()
    tmin = a[kept].min()
    assert float(tmin) >= float(a[~kept].max())
    ties = (a == tmin).nonzero().flatten()
    n_taken = int(kept[ties].sum())
    assert bool(kept[ties[:n_taken]].all()) and not bool(kept[ties[n_taken:]].any())
    del kept, a, x, v, i
    torch.cuda.empty_cache()


def test_workspace_too_small_is_rejected(mpc):
    L = 100003
    need = mpc.mpc_topk_workspace_bytes(1, L, 10)
    assert need > 0
    x = torch.zeros((1, L), device="cuda")
    ws = torch.empty(need - 256, dtype=torch.uint8, device="cuda")
    with pytest.raises(mpc.MpcError) as e:
        mpc.mpc_topk_compress(x, 10, ws=ws)
    assert e.value.status == 3


@pytest.mark.parametrize("L", [131072, 1000003])
def test_sample_misled(mpc, L):
    """A row with 16384 evenly spread magnitudes much larger than the rest, which the
    evenly spread sample over-represents: the sampled band misses the k-th entry after the
    first read, and the multi-pass path finishes the selection (error feedback: with s
    already written into err).  Plain, EF and EF21, against the oracle."""
    rng = np.random.default_rng(L)
    R = 1
    x = (rng.standard_normal((R, L)) * 1e-3).astype(np.float32)
    pos = (np.arange(16384, dtype=np.int64) * L) // 16384
    x[0, pos] = (1.0 + rng.random(16384)).astype(np.float32)
    k = L // 4  # far more than the sampled entries: the threshold is among the small ones
    v, i = mpc.mpc_topk_compress(dev(x), k)
    ok(mpc)
    ov, oi = oracle.topk_compress(x, k)
    assert_bits_equal(i.cpu().numpy(), oi, "idx")
    assert_bits_equal(v.cpu().numpy(), ov, "vals")
    e_host = (rng.standard_normal((R, L)) * 1e-4).astype(np.float32)
    e_dev = dev(e_host.copy())
    v, i = mpc.mpc_ef_topk_compress(dev(x), e_dev, k)
    ok(mpc)
    ov, oi = oracle.ef_topk_compress(x, e_host, k)
    assert_bits_equal(i.cpu().numpy(), oi, "EF idx")
    assert_bits_equal(v.cpu().numpy(), ov, "EF vals")
    assert_bits_equal(e_dev.cpu().numpy(), e_host, "EF err")
    g_host = (rng.standard_normal((R, L)) * 1e-4).astype(np.float32)
    g_dev = dev(g_host.copy())
    v, i = mpc.mpc_ef21_topk_compress(dev(x), g_dev, k)
    ok(mpc)
    ov, oi = oracle.ef21_topk_compress(x, g_host, k)
    assert_bits_equal(i.cpu().numpy(), oi, "EF21 idx")
    assert_bits_equal(g_dev.cpu().numpy(), g_host, "EF21 g")


@pytest.mark.parametrize("R,L", [(70, 70000), (9, 131073), (3, 1 << 20)])
def test_many_long_rows(mpc, R, L):
    """Several long rows in one call: the grid path takes up to 64 rows a batch (the row
    in blockIdx.y, a workspace slice each), so 70 rows make a full batch and a partial
    one.  Plain TopK at K = 1 / 10 / 50 % and two steps of error feedback, every row
    against the oracle."""
    rng = np.random.default_rng(7 * R + L)
    x = rng.standard_normal((R, L)).astype(np.float32)
    for k in sorted({max(1, L // 100), L // 10, L // 2}):
        v, i = mpc.mpc_topk_compress(dev(x), k)
        ok(mpc)
        ov, oi = oracle.topk_compress(x, k)
        assert_bits_equal(i.cpu().numpy(), oi, "idx R=%d L=%d k=%d" % (R, L, k))
        assert_bits_equal(v.cpu().numpy(), ov, "vals R=%d L=%d k=%d" % (R, L, k))
    k = L // 10
    e_host = np.zeros((R, L), np.float32)
    e_dev = torch.zeros((R, L), device="cuda")
    for step in range(2):
        v, i = mpc.mpc_ef_topk_compress(dev(x), e_dev, k)
        ok(mpc)
        ov, oi = oracle.ef_topk_compress(x, e_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "EF vals step %d" % step)
        assert_bits_equal(e_dev.cpu().numpy(), e_host, "EF err step %d" % step)
        x = (x + 0.1 * rng.standard_normal((R, L))).astype(np.float32)


def test_long_rows_of_every_kind_in_one_batch(mpc):
    """One batch whose rows take different paths: rows the sampled band resolves next to
    rows of equal values, zeros and few distinct magnitudes, and a row whose sampled
    positions hold the largest magnitudes, which fall back to the multi-pass path.  Every
    row against the oracle, plain and with error feedback."""
    L = 100000
    rows = [rows_of(kind, 1, L, seed=11 + n)[0].astype(np.float32) for n, kind in enumerate(KINDS)]
    rng = np.random.default_rng(5)
    misled = (rng.standard_normal(L) * 1e-3).astype(np.float32)
    pos = (np.arange(1024, dtype=np.int64) * L) // 1024  # the sample of a row this long
    misled[pos] = (1.0 + rng.random(1024)).astype(np.float32)
    x = np.stack(rows + [misled])
    R = x.shape[0]
    for k in (L // 100, L // 4):
        v, i = mpc.mpc_topk_compress(dev(x), k)
        ok(mpc)
        ov, oi = oracle.topk_compress(x, k)
        assert_bits_equal(i.cpu().numpy(), oi, "idx k=%d" % k)
        assert_bits_equal(v.cpu().numpy(), ov, "vals k=%d" % k)
        e_host = (rng.standard_normal((R, L)) * 1e-4).astype(np.float32)
        e_dev = dev(e_host.copy())
        v, i = mpc.mpc_ef_topk_compress(dev(x), e_dev, k)
        ok(mpc)
        ov, oi = oracle.ef_topk_compress(x, e_host, k)
        assert_bits_equal(i.cpu().numpy(), oi, "EF idx k=%d" % k)
        assert_bits_equal(v.cpu().numpy(), ov, "EF vals k=%d" % k)
        assert_bits_equal(e_dev.cpu().numpy(), e_host, "EF err k=%d" % k)
