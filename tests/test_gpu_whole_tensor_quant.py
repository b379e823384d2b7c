"""Whole-tensor quantisation (§2.2 applied to a whole tensor as one row, the last row
length of the bandwidth sweep): a single row of 2^27 .. 2^30 entries takes the two-pass
path (row extrema in a caller workspace, then the coding kernel), with 64-bit code and
bit offsets.  Every code word, the scale and the minimum are compared bit for bit with
the CPU oracle on the whole row; dequantised values on the whole row at 2^28 and on
ranges at the start, middle and end of the 2^30 row."""

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


@pytest.fixture(scope="module")
def synth():
    from paper_2401_07788_gb300 import synth as s

    return s


def ok(mpc):
    assert mpc.mpc_get_status() == 0, mpc.mpc_last_error()


def check_row(mpc, x, bits, sr, seed, dequant=True):
    N = x.numel()
    xr = x.view(1, N)
    cq, sq, mq = mpc.mpc_quant_compress(xr, bits, stochastic=sr, seed=seed)
    ok(mpc)
    xn = xr.cpu().numpy()
    oc, os_, om = oracle.quant_compress(xn, bits, sr, seed)
    tag = "N=%d bits=%d sr=%d" % (N, bits, sr)
    assert_bits_equal(cq.cpu().numpy().view(np.uint32), oc, "codes " + tag)
    assert_bits_equal(sq.cpu().numpy(), os_, "scale " + tag)
    assert_bits_equal(mq.cpu().numpy(), om, "minv " + tag)
    if dequant:
        y = mpc.mpc_quant_decompress(cq, sq, mq, N, bits)
        ok(mpc)
        assert_bits_equal(y.cpu().numpy(), oracle.quant_decompress(oc, os_, om, N, bits),
                          "dequant " + tag)
        del y
    del cq


@pytest.mark.parametrize("bits,sr", [(2, False), (4, False), (8, False), (6, False),
                                     (4, True), (2, True)])
def test_whole_row_2p28(mpc, synth, bits, sr):
    x = synth.normal((1 << 28,), 28, "cuda")
    check_row(mpc, x, bits, sr, (5 << 32) | 3)
    del x
    torch.cuda.empty_cache()


@pytest.mark.parametrize("bits,sr", [(6, False), (2, True)])
def test_whole_row_ragged(mpc, synth, bits, sr):
    """A row of 2^27 + 12345 entries: not a multiple of 4 (plain loads, no bulk copies) and
    a partial last slice."""
    x = synth.normal(((1 << 27) + 12345,), 27, "cuda")
    check_row(mpc, x, bits, sr, 11)
    del x
    torch.cuda.empty_cache()


def test_whole_row_2p30(mpc, synth):
    """One row of 2^30 entries (4 GiB), 8-bit nearest: every code word, scale and minimum;
    dequantised values on three ranges of 2^20 entries."""
    N = 1 << 30
    bits = 8
    x = synth.normal((N,), 30, "cuda").view(1, N)
    cq, sq, mq = mpc.mpc_quant_compress(x, bits)
    ok(mpc)
    xn = x.cpu().numpy()
    oc, os_, om = oracle.quant_compress(xn, bits)
    del xn
    got = cq.cpu().numpy().view(np.uint32)
    assert_bits_equal(got, oc, "codes")
    assert_bits_equal(sq.cpu().numpy(), os_, "scale")
    assert_bits_equal(mq.cpu().numpy(), om, "minv")
    y = mpc.mpc_quant_decompress(cq, sq, mq, N, bits)
    ok(mpc)
    n = 1 << 20
    per_word = 32 // bits
    for a in (0, N // 2 + 4096, N - n):
        words = oc[0, a // per_word:(a + n) // per_word][None, :]
        want = oracle.quant_decompress(words, os_, om, n, bits)
        assert_bits_equal(y[0, a:a + n].cpu().numpy()[None, :], want, "dequant at %d" % a)
    del x, cq, y
    torch.cuda.empty_cache()
