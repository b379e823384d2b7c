"""TopK index reuse (§3.2, Table 5) on the GPU through the C ABI against the CPU oracle,
bit for bit: the gradient's values at the activation's payload indices, and the round
trip through decompression."""

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
    return m


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def ok(mpc):
    assert mpc.mpc_get_status() == 0, mpc.mpc_last_error()


@pytest.mark.parametrize("L", [1, 7, 128, 769, 4096, 4099, 32768, 65536, 100003])
def test_gather_at_activation_indices(mpc, L):
    """The backward of a boundary: gradient values at the forward's kept indices."""
    R = 5
    a = rows_of("relu", R, L, seed=L)
    g = rows_of("normal", R, L, seed=L + 1)
    for k in sorted({1, max(1, L // 10), max(1, L // 3), L}):
        _, idx = oracle.topk_compress(a, k)
        v = mpc.mpc_topk_gather(dev(g), dev(idx))
        ok(mpc)
        assert_bits_equal(v.cpu().numpy(), oracle.topk_gather(g, idx), "vals L=%d k=%d" % (L, k))
        y = mpc.mpc_topk_decompress(v, dev(idx), L)
        ok(mpc)
        want = oracle.topk_decompress(oracle.topk_gather(g, idx), idx, L)
        assert_bits_equal(y.cpu().numpy(), want, "round trip L=%d k=%d" % (L, k))


@pytest.mark.parametrize("kind", KINDS)
def test_gather_kinds(mpc, kind):
    R, L, k = 3, 3000, 301
    g = rows_of(kind, R, L, seed=11)
    idx = np.sort(np.random.default_rng(12).permuted(np.tile(np.arange(L), (R, 1)), axis=1)[:, :k],
                  axis=1).astype(np.int32)
    v = mpc.mpc_topk_gather(dev(g), dev(idx))
    ok(mpc)
    assert_bits_equal(v.cpu().numpy(), oracle.topk_gather(g, idx), kind)


def test_gather_unaligned_and_any_order(mpc):
    """Payload rows that do not start on 16 bytes (k % 4 != 0, offset views) and indices
    in no particular order."""
    R, L, k = 7, 1001, 333
    g = rows_of("heavy", R, L, seed=21)
    rng = np.random.default_rng(22)
    idx = np.stack([rng.permutation(L)[:k] for _ in range(R)]).astype(np.int32)
    base = torch.zeros(R * k + 1, dtype=torch.int32, device="cuda")
    idx_dev = base[1:].view(R, k)
    idx_dev.copy_(dev(idx))
    out = torch.zeros(R * k + 1, device="cuda")[1:].view(R, k)
    mpc.mpc_topk_gather(dev(g), idx_dev, vals=out)
    ok(mpc)
    assert_bits_equal(out.cpu().numpy(), oracle.topk_gather(g, idx), "unaligned")


def test_gather_cnn_boundary_full(mpc):
    """The CNN stage boundary (128 x 32768), K = 10 %, every row."""
    from paper_2401_07788_gb300 import synth

    R, L = 128, 32768
    k = synth.k_of(L, 10)
    a = synth.relu_normal((R, L), 0, "cuda")
    g = synth.normal((R, L), 1, "cuda", std=1e-3)
    _, idx = mpc.mpc_topk_compress(a, k)
    v = mpc.mpc_topk_gather(g, idx)
    ok(mpc)
    gn, ixn = g.cpu().numpy(), idx.cpu().numpy()
    assert_bits_equal(v.cpu().numpy(), oracle.topk_gather(gn, ixn), "cnn boundary")


def test_gather_bad_index_is_reported(mpc):
    R, L, k = 2, 64, 8
    g = rows_of("normal", R, L, seed=31)
    idx = np.tile(np.arange(0, 64, 8, dtype=np.int32), (R, 1))
    idx[1, 3] = L  # out of range
    v = mpc.mpc_topk_gather(dev(g), dev(idx))
    assert mpc.mpc_get_status() == 6  # MPC_ERR_DEVICE
    vv = v.cpu().numpy()
    assert vv[1, 3] == 0.0
    good = idx.copy()
    good[1, 3] = 0
    want = oracle.topk_gather(g, good)
    want[1, 3] = 0.0
    assert_bits_equal(vv, want, "other entries")
    ok(mpc)  # the status word was cleared by the read
