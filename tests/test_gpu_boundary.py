"""The compression block between pipeline stages (§2.1, Figure 1) on the GPU: its forward
output and its backward gradient against the CPU oracle's compress-then-decompress, bit
for bit, for every compressor, over several steps of feedback state; the inference
switch; a pipeline of four stages with three blocks."""

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


def k_of(L, pct):
    return max(1, L * pct // 100)


def run(block, x, gy, ids=None):
    xx = x.clone().requires_grad_(True)
    y = block(xx, ids) if ids is not None else block(xx)
    y.backward(gy)
    torch.cuda.synchronize()
    return y.detach(), xx.grad


def orc_topk(a, pct):
    v, i = oracle.topk_compress(a, k_of(a.shape[1], pct))
    return oracle.topk_decompress(v, i, a.shape[1]), i


def test_topk_both_directions(mpc):
    B = mpc.CompressionBoundary(mpc.TopK(10), mpc.TopK(30))
    x = torch.randn(8, 4, 8, 8, device="cuda")
    gy = torch.randn_like(x)
    y, gx = run(B, x, gy)
    want_y, _ = orc_topk(x.cpu().numpy().reshape(8, -1), 10)
    want_g, _ = orc_topk(gy.cpu().numpy().reshape(8, -1), 30)
    assert_bits_equal(y.cpu().numpy().reshape(8, -1), want_y, "activation")
    assert_bits_equal(gx.cpu().numpy().reshape(8, -1), want_g, "gradient")


def test_index_reuse(mpc):
    """Gradients at the activation's kept indices (§3.2, Table 5)."""
    B = mpc.CompressionBoundary(mpc.TopK(20), mpc.Reuse())
    x = torch.randn(6, 300, device="cuda")
    gy = torch.randn_like(x)
    y, gx = run(B, x, gy)
    xn, gn = x.cpu().numpy(), gy.cpu().numpy()
    want_y, idx = orc_topk(xn, 20)
    want_g = oracle.topk_decompress(oracle.topk_gather(gn, idx), idx, 300)
    assert_bits_equal(y.cpu().numpy(), want_y, "activation")
    assert_bits_equal(gx.cpu().numpy(), want_g, "gradient")


@pytest.mark.parametrize("fb", ["ef", "ef21"])
def test_feedback_over_steps(mpc, fb):
    B = mpc.CompressionBoundary(mpc.TopK(10, feedback=fb), None)
    state = np.zeros((4, 512), np.float32)
    rng = np.random.default_rng(0)
    for step in range(4):
        xn = rng.standard_normal((4, 512)).astype(np.float32)
        y, gx = run(B, torch.from_numpy(xn).cuda(), torch.ones(4, 512, device="cuda"))
        k = k_of(512, 10)
        f = oracle.ef_topk_compress if fb == "ef" else oracle.ef21_topk_compress
        v, i = f(xn, state, k)
        # EF's receiver takes the message; EF21's takes its copy of g' = g + C(x - g)
        want = oracle.topk_decompress(v, i, 512) if fb == "ef" else state
        assert_bits_equal(y.cpu().numpy(), want, "%s step %d" % (fb, step))
        assert_bits_equal(B.state.cpu().numpy(), state, "%s state step %d" % (fb, step))
        assert torch.equal(gx, torch.ones_like(gx))  # no gradient compressor


def test_aqsgd_per_sample_buffer(mpc):
    S, rps, L = 10, 3, 256
    B = mpc.CompressionBoundary(mpc.TopK(30, feedback="aqsgd"), mpc.TopK(30), rows="last",
                                aqsgd_samples=S)
    buf = np.zeros((S, rps, L), np.float32)
    rng = np.random.default_rng(1)
    for step in range(3):
        ids = rng.permutation(S)[:4].astype(np.int64)
        xn = rng.standard_normal((4, rps, L)).astype(np.float32)
        y, _ = run(B, torch.from_numpy(xn).cuda(), torch.zeros(4, rps, L, device="cuda"),
                   torch.from_numpy(ids).cuda())
        oracle.aqsgd_compress(xn, buf, ids, k_of(L, 30))
        # the next stage receives its copy of the samples' updated buffer rows
        assert_bits_equal(y.cpu().numpy(), buf[ids], "aqsgd step %d" % step)
        assert_bits_equal(B.state.cpu().numpy(), buf, "buffer step %d" % step)


@pytest.mark.parametrize("bits,sr", [(4, False), (8, True)])
def test_aqsgd_quant_per_sample_buffer(mpc, bits, sr):
    """AQ-SGD with the quantiser (§2.5's cited work): the change against each sample's
    buffer is quantised; the next stage receives the updated buffer rows."""
    S, L = 12, 2 * 8 * 8
    B = mpc.CompressionBoundary(mpc.Quant(bits, sr, feedback="aqsgd"), mpc.Quant(8),
                                aqsgd_samples=S, seed=3)
    buf = np.zeros((S, 1, L), np.float32)
    rng = np.random.default_rng(2)
    base = rng.standard_normal((S, 2, 8, 8)).astype(np.float32)
    for step in range(3):
        ids = rng.permutation(S)[:5].astype(np.int64)
        xn = (base[ids] + 0.1 * rng.standard_normal((5, 2, 8, 8))).astype(np.float32)
        gn = rng.standard_normal((5, 2, 8, 8)).astype(np.float32)
        y, gx = run(B, torch.from_numpy(xn).cuda(), torch.from_numpy(gn).cuda(),
                    torch.from_numpy(ids).cuda())
        seed_fw = (((3 << 1) | 0) << 32) | step
        oracle.aqsgd_quant_compress(xn.reshape(5, 1, L), buf, ids, bits, sr, seed_fw)
        assert_bits_equal(y.cpu().numpy().reshape(5, 1, L), buf[ids], "aqsgd-q step %d" % step)
        assert_bits_equal(B.state.cpu().numpy(), buf, "buffer step %d" % step)
        c, s_, m = oracle.quant_compress(gn.reshape(5, L), 8, False, 0)
        assert_bits_equal(gx.cpu().numpy().reshape(5, L),
                          oracle.quant_decompress(c, s_, m, L, 8), "gradient step %d" % step)


@pytest.mark.parametrize("bits,sr", [(2, False), (4, True), (6, False), (8, True)])
def test_quant_both_directions(mpc, bits, sr):
    B = mpc.CompressionBoundary(mpc.Quant(bits, sr), mpc.Quant(bits, sr), rows="last", seed=5)
    x = torch.randn(2, 16, 96, device="cuda")
    gy = torch.randn_like(x) * 1e-3
    y, gx = run(B, x, gy)
    seed_fw = (((5 << 1) | 0) << 32) | 0
    seed_bw = (((5 << 1) | 1) << 32) | 1  # the step counter has advanced by the backward
    xn = x.cpu().numpy().reshape(-1, 96)
    gn = gy.cpu().numpy().reshape(-1, 96)
    c, s, m = oracle.quant_compress(xn, bits, sr, seed_fw)
    assert_bits_equal(y.cpu().numpy().reshape(-1, 96), oracle.quant_decompress(c, s, m, 96, bits), "fw")
    c, s, m = oracle.quant_compress(gn, bits, sr, seed_bw)
    assert_bits_equal(gx.cpu().numpy().reshape(-1, 96), oracle.quant_decompress(c, s, m, 96, bits), "bw")


def test_inference_switch(mpc):
    x = torch.randn(4, 100, device="cuda")
    off = mpc.CompressionBoundary(mpc.TopK(10, feedback="ef"), mpc.TopK(10)).eval()
    assert off(x) is x
    on = mpc.CompressionBoundary(mpc.TopK(10, feedback="ef"), mpc.TopK(10),
                                 compress_at_inference=True)
    on.train()
    on(x.clone())
    state = on.state.clone()
    on.eval()
    y = on(x)
    want, _ = orc_topk(x.cpu().numpy(), 10)  # plain TopK: no feedback at inference
    assert_bits_equal(y.cpu().numpy(), want, "inference")
    assert torch.equal(on.state, state)


def test_pipeline_of_four_stages(mpc):
    """Model-parallel degree 4 (§3.2): three blocks between four stages; one training step
    runs through every block in both directions."""
    torch.manual_seed(0)
    stages = [torch.nn.Sequential(torch.nn.Linear(64, 64), torch.nn.ReLU()) for _ in range(3)]
    stages.append(torch.nn.Linear(64, 10))
    model = mpc.with_boundaries(stages, lambda i: mpc.CompressionBoundary(
        mpc.TopK(30, feedback="ef21"), mpc.Reuse())).cuda()
    assert sum(isinstance(m, mpc.CompressionBoundary) for m in model) == 3
    x = torch.randn(32, 64, device="cuda")
    t = torch.randint(0, 10, (32,), device="cuda")
    opt = torch.optim.SGD(model.parameters(), lr=0.1)
    losses = []
    for _ in range(30):
        opt.zero_grad()
        loss = torch.nn.functional.cross_entropy(model(x), t)
        loss.backward()
        opt.step()
        losses.append(float(loss.detach()))
    assert mpc.mpc_get_status() == 0, mpc.mpc_last_error()
    assert all(p.grad is not None for p in model.parameters())
    assert losses[-1] < losses[0]
