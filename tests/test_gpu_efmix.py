"""EF-mixed TopK (§2.4) on the GPU through the C ABI against the CPU oracle, bit for bit
(payload, indices and the error buffer over several steps), at reduced and full sizes,
on the on-chip and multi-pass paths."""

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


def steps(mpc, x0, k, n_steps, seed, drift=0.3):
    rng = np.random.default_rng(seed)
    R, L = x0.shape
    e_host = np.zeros((R, L), np.float32)
    e_dev = torch.zeros((R, L), device="cuda")
    x = x0
    for step in range(n_steps):
        v, i = mpc.mpc_efmix_topk_compress(dev(x), e_dev, k)
        assert mpc.mpc_get_status() == 0, mpc.mpc_last_error()
        ov, oi = oracle.efmix_topk_compress(x, e_host, k)
        tag = "L=%d k=%d step %d" % (L, k, step)
        assert_bits_equal(i.cpu().numpy(), oi, "idx " + tag)
        assert_bits_equal(v.cpu().numpy(), ov, "vals " + tag)
        assert_bits_equal(e_dev.cpu().numpy(), e_host, "err " + tag)
        x = (x + drift * rng.standard_normal((R, L))).astype(np.float32)


@pytest.mark.parametrize("L", [1, 2, 7, 128, 769, 1024, 2049, 4096, 8193, 32768, 65536])
def test_efmix_lengths(mpc, L):
    x = rows_of("normal", 3, L, seed=L)
    for k in sorted({1, min(2, L), max(1, L // 10), max(1, L // 3), L}):
        steps(mpc, x, k, 3, seed=k)


@pytest.mark.parametrize("kind", KINDS)
def test_efmix_kinds(mpc, kind):
    x = rows_of(kind, 4, 3000, seed=7)
    steps(mpc, x, 300, 3, seed=8, drift=0.0 if kind in ("zeros", "equal", "ties") else 0.3)


def test_efmix_cnn_boundary(mpc):
    """The CNN stage boundary, Top10 %, ReLU activations drifting step to step."""
    from paper_2401_07788_gb300 import synth

    R, L = 128, 32768
    x = synth.relu_normal((R, L), 0, "cpu").numpy()
    steps(mpc, x, synth.k_of(L, 10), 2, seed=3, drift=0.1)


def test_efmix_multipass_path(mpc):
    """Rows longer than a cluster holds, and the forced multi-pass path."""
    steps(mpc, rows_of("normal", 2, 100003, seed=1), 10000, 2, seed=2)
    mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, 2)
    try:
        steps(mpc, rows_of("relu", 2, 5000, seed=4), 500, 2, seed=5)
    finally:
        mpc.mpc_set_knob(mpc.MPC_KNOB_TOPK_PATH, 0)


def test_efmix_workspace_is_required(mpc):
    R, L, k = 2, 1000, 100
    need = mpc.mpc_efmix_workspace_bytes(R, L, k)
    assert need > 0
    x = torch.zeros((R, L), device="cuda")
    e = torch.zeros_like(x)
    ws = torch.empty(need - 256, dtype=torch.uint8, device="cuda")
    with pytest.raises(mpc.MpcError) as ex:
        mpc.mpc_efmix_topk_compress(x, e, k, ws=ws)
    assert ex.value.status == 3
