"""The five stage-boundary workloads at their full sizes, in the launch configuration the
benchmark uses, against the CPU oracle: every output where the oracle finishes in seconds,
sampled rows (recomputed one by one by the oracle) where it does not."""

import numpy as np
import pytest
import torch

import oracle
from gpu_cases import assert_bits_equal, row_blocks

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def mpc():
    import __graft_entry__ as g

    g.build()
    import paper_2401_07788_gb300 as m

    torch.cuda.set_device(0)
    return m


@pytest.fixture(scope="module")
def synth():
    from paper_2401_07788_gb300 import synth as s

    return s


def ok(mpc):
    assert mpc.mpc_get_status() == 0, mpc.mpc_last_error()


def test_cnn_small_boundary(mpc, synth):
    """ResNet-18 boundary [32,64,16,16]: Top10% of the activation, 8-bit gradient."""
    c = synth.CNN_SMALL
    x = synth.relu_normal(c["shape"], 0, "cuda").view(c["rows"], c["row_len"])
    g = synth.normal(c["shape"], 1, "cuda", std=1e-3).view(c["rows"], c["row_len"])
    k = synth.k_of(c["row_len"], c["topk_percent"])
    v, i = mpc.mpc_topk_compress(x, k)
    y = mpc.mpc_topk_decompress(v, i, c["row_len"])
    cq, sq, mq = mpc.mpc_quant_compress(g, 8)
    gy = mpc.mpc_quant_decompress(cq, sq, mq, c["row_len"], 8)
    ok(mpc)
    xn, gn = x.cpu().numpy(), g.cpu().numpy()
    ov, oi = oracle.topk_compress(xn, k)
    assert_bits_equal(i.cpu().numpy(), oi, "idx")
    assert_bits_equal(v.cpu().numpy(), ov, "vals")
    assert_bits_equal(y.cpu().numpy(), oracle.topk_decompress(ov, oi, c["row_len"]), "y")
    oc, os_, om = oracle.quant_compress(gn, 8)
    assert_bits_equal(cq.cpu().numpy().view(np.uint32), oc, "codes")
    assert_bits_equal(gy.cpu().numpy(), oracle.quant_decompress(oc, os_, om, c["row_len"], 8),
                      "dequant")


@pytest.mark.parametrize("seed", [0, 9])
def test_cnn_boundary_ef_and_quant(mpc, synth, seed):
    """[128,128,16,16] for all 50 steps of the workload: EF-TopK at 5/10/30% with the
    error carried over the drifting steps, and 2/4/8-bit gradients, nearest and stochastic
    (seed (config_seed << 32) | step); every output compared at every step."""
    c = synth.CNN
    R, L = c["rows"], c["row_len"]
    gen = synth.generator(seed, "cuda")
    x = synth.relu_normal(c["shape"], seed, "cuda", gen=gen).view(R, L)
    errs = {p: torch.zeros((R, L), device="cuda") for p in c["topk_percents"]}
    errs_host = {p: np.zeros((R, L), np.float32) for p in c["topk_percents"]}
    for step in range(c["steps"]):
        xn = x.cpu().numpy()
        for p in c["topk_percents"]:
            k = synth.k_of(L, p)
            v, i = mpc.mpc_ef_topk_compress(x, errs[p], k)
            ok(mpc)
            ov, oi = row_blocks(lambda xb, eb: oracle.ef_topk_compress(xb, eb, k), R, xn,
                                errs_host[p])
            assert_bits_equal(i.cpu().numpy(), oi, "idx K=%d step %d" % (p, step))
            assert_bits_equal(v.cpu().numpy(), ov, "vals K=%d step %d" % (p, step))
            assert_bits_equal(errs[p].cpu().numpy(), errs_host[p], "err K=%d step %d" % (p, step))
        g = synth.normal((R, L), 1000 * seed + step, "cuda", std=1e-3)
        gn = g.cpu().numpy()
        for bits in c["bits"]:
            for sr in (False, True):
                sd = (seed << 32) | step
                cq, sq, mq = mpc.mpc_quant_compress(g, bits, stochastic=sr, seed=sd)
                ok(mpc)
                if sr:
                    oc, os_, om = oracle.quant_compress(gn, bits, sr, sd)
                else:
                    oc, os_, om = row_blocks(lambda gb: oracle.quant_compress(gb, bits), R, gn)
                what = "b=%d sr=%d step %d" % (bits, sr, step)
                assert_bits_equal(cq.cpu().numpy().view(np.uint32), oc, "codes " + what)
                assert_bits_equal(sq.cpu().numpy(), os_, "scale " + what)
                assert_bits_equal(mq.cpu().numpy(), om, "minv " + what)
        x = synth.drift(x, c["drift"], gen)


def test_lm_boundary_ef21_and_quant(mpc, synth):
    """GPT-2 boundary [8,1024,768] with outlier channels, all 20 steps of the workload:
    EF21-TopK 10% per token, g_0 = 0, over drifting steps, and 4-bit per-token gradient
    quantisation of each step's gradient."""
    c = synth.LM
    R, L = c["rows"], c["row_len"]
    k = synth.k_of(L, c["topk_percent"])
    x = synth.lm_hidden(0, "cuda")
    gen = synth.generator(1, "cuda")
    g_dev = torch.zeros((R, L), device="cuda")
    g_host = np.zeros((R, L), np.float32)
    for step in range(c["steps"]):
        xn = x.cpu().numpy()
        v, i = mpc.mpc_ef21_topk_compress(x, g_dev, k)
        ok(mpc)
        ov, oi = row_blocks(lambda xb, gb: oracle.ef21_topk_compress(xb, gb, k), R, xn, g_host)
        assert_bits_equal(i.cpu().numpy(), oi, "idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "vals step %d" % step)
        assert_bits_equal(g_dev.cpu().numpy(), g_host, "g step %d" % step)
        gr = synth.normal((R, L), 2 + step, "cuda", std=1e-4)
        cq, sq, mq = mpc.mpc_quant_compress(gr, 4)
        y = mpc.mpc_quant_decompress(cq, sq, mq, L, 4)
        ok(mpc)
        oc, os_, om = row_blocks(lambda gb: oracle.quant_compress(gb, 4), R, gr.cpu().numpy())
        assert_bits_equal(cq.cpu().numpy().view(np.uint32), oc, "codes step %d" % step)
        assert_bits_equal(y.cpu().numpy(), oracle.quant_decompress(oc, os_, om, L, 4),
                          "dequant step %d" % step)
        x = synth.drift(x, c["drift"], gen)


def test_aqsgd_boundary_full_buffer(mpc, synth):
    """Per-sample buffer [4096,512,1024] (2^31 entries, 64-bit offsets), 10 steps of 16 ids,
    Top30% of the change: the gathered rows are checked against the oracle at every step,
    the receiver's copy of the buffer (updated from the payload alone) stays bit-identical
    to the sender's, and rows of samples not drawn stay bit-identical."""
    c = synth.AQSGD
    S, rps, L = c["num_samples"], c["rows_per_sample"], c["row_len"]
    k = synth.k_of(L, c["topk_percent"])
    buf = synth.normal((S, rps, L), 0, "cuda")
    recv = buf.clone()
    watch = torch.tensor([0, 1, S // 2, S - 1], device="cuda")
    gen = synth.generator(5, "cuda")
    n = c["ids_per_step"]
    for step in range(10):
        ids = synth.sample_ids(S, n, 100 + step, "cuda")
        x = buf[ids] + c["noise"] * torch.randn((n, rps, L), generator=gen, device="cuda")
        rows_before = buf[ids].cpu().numpy()
        untouched = watch[~torch.isin(watch, ids)]
        keep = buf[untouched].clone()
        v, i = mpc.mpc_aqsgd_compress(x, buf, ids, k)
        mpc.mpc_aqsgd_decompress(v, i, recv, ids)
        ok(mpc)
        local = rows_before.copy()
        ov, oi = row_blocks(
            lambda xb, lb: oracle.aqsgd_compress(xb, lb, np.arange(xb.shape[0]), k), n,
            x.cpu().numpy(), local)
        assert_bits_equal(i.cpu().numpy(), oi, "idx step %d" % step)
        assert_bits_equal(v.cpu().numpy(), ov, "vals step %d" % step)
        assert_bits_equal(buf[ids].cpu().numpy(), local, "buffer rows step %d" % step)
        assert torch.equal(recv[ids].view(torch.int32), buf[ids].view(torch.int32)), step
        assert torch.equal(buf[untouched], keep)
    assert torch.equal(recv.view(torch.int32), buf.view(torch.int32))
    del buf, recv
    torch.cuda.empty_cache()


@pytest.mark.parametrize("log2n", [20, 26, 30])
@pytest.mark.parametrize("L", [768, 4096, 65536])
def test_sweep_sampled_rows(mpc, synth, log2n, L):
    """Single N(0,1) tensors of 2^20..2^30 entries as rows of L: TopK 1/10/50% plain and
    with error feedback, 2/4/8-bit quantisation; 8 sampled rows recomputed by the oracle."""
    N = 1 << log2n
    R = N // L
    x = synth.normal((R * L,), log2n, "cuda").view(R, L)
    rows = np.unique(np.random.default_rng(log2n + L).integers(0, R, 8))
    rows = np.unique(np.concatenate([rows, [0, R - 1]]))
    xs = x[torch.from_numpy(rows).cuda()].cpu().numpy()
    for pct in (1, 10, 50):
        k = synth.k_of(L, pct)
        v, i = mpc.mpc_topk_compress(x, k)
        ok(mpc)
        ov, oi = oracle.topk_compress(xs, k)
        assert_bits_equal(i[rows].cpu().numpy(), oi, "idx K=%d" % pct)
        assert_bits_equal(v[rows].cpu().numpy(), ov, "vals K=%d" % pct)
        del v, i
        err = torch.full_like(x, 0.25)
        v, i = mpc.mpc_ef_topk_compress(x, err, k)
        ok(mpc)
        eh = np.full_like(xs, 0.25)
        ov, oi = oracle.ef_topk_compress(xs, eh, k)
        assert_bits_equal(i[rows].cpu().numpy(), oi, "EF idx K=%d" % pct)
        assert_bits_equal(err[rows].cpu().numpy(), eh, "EF err K=%d" % pct)
        del v, i, err
    for bits in (2, 4, 8):
        cq, sq, mq = mpc.mpc_quant_compress(x, bits)
        ok(mpc)
        oc, os_, om = oracle.quant_compress(xs, bits)
        assert_bits_equal(cq[rows].cpu().numpy().view(np.uint32), oc, "codes b=%d" % bits)
        assert_bits_equal(sq[rows].cpu().numpy(), os_, "scale b=%d" % bits)
    del x
    torch.cuda.empty_cache()


def rel_err(x, y) -> float:
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    return float(np.linalg.norm(x - y) / np.linalg.norm(x))


def test_compression_error_norms(mpc, synth):
    """Relative compression error ||x - x_hat|| / ||x|| (computed in double) of every
    operator on the CNN boundary: the GPU's within 1e-6 relative of the oracle's (they are
    bit-identical, so the norms agree exactly), and each one inside the range its
    operator allows (TopK below the energy of the dropped tail; b-bit quantisation below
    half a step per entry)."""
    c = synth.CNN
    R, L = c["rows"], c["row_len"]
    x = synth.relu_normal(c["shape"], 3, "cuda").view(R, L)
    xn = x.cpu().numpy()
    for p in c["topk_percents"]:
        k = synth.k_of(L, p)
        v, i = mpc.mpc_topk_compress(x, k)
        y = mpc.mpc_topk_decompress(v, i, L)
        ok(mpc)
        ov, oi = oracle.topk_compress(xn, k)
        e_gpu = rel_err(xn, y.cpu().numpy())
        e_orc = rel_err(xn, oracle.topk_decompress(ov, oi, L))
        assert abs(e_gpu - e_orc) <= 1e-6 * e_orc
        # the dropped entries are the L - k smallest magnitudes of each row
        srt = np.sort(np.abs(xn.astype(np.float64)), axis=1)[:, : L - k]
        assert abs(e_gpu - np.sqrt((srt ** 2).sum()) / np.linalg.norm(xn.astype(np.float64))) <= 1e-9
    g = synth.normal((R, L), 77, "cuda", std=1e-3)
    gn = g.cpu().numpy()
    for bits in c["bits"]:
        for sr in (False, True):
            cq, sq, mq = mpc.mpc_quant_compress(g, bits, stochastic=sr, seed=5)
            y = mpc.mpc_quant_decompress(cq, sq, mq, L, bits)
            ok(mpc)
            oc, os_, om = oracle.quant_compress(gn, bits, sr, 5)
            e_gpu = rel_err(gn, y.cpu().numpy())
            e_orc = rel_err(gn, oracle.quant_decompress(oc, os_, om, L, bits))
            assert abs(e_gpu - e_orc) <= 1e-6 * e_orc
            # nearest: |x - y| <= scale / 2 (+ rounding); stochastic: < scale
            bound = (0.5 if not sr else 1.0) * np.asarray(os_, np.float64) * np.sqrt(L) * 1.0001
            rows = np.linalg.norm(gn.astype(np.float64) - y.cpu().numpy(), axis=1)
            assert (rows <= bound).all(), "b=%d sr=%d" % (bits, sr)
