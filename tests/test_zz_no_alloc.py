"""mpc_quant_compress_noalloc, the quantisation entry point for callers that cannot
allocate device memory (its per-row scratch is a static device array), gives the same
codes, scales and minima as mpc_quant_compress, bit for bit, on two calls in a row.

The test calls both entry points through the C ABI (ctypes, raw device pointers).  It is
kept in a file of its own that pytest collects last."""

import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__ as g

    g.build()
    import paper_2401_07788_gb300 as mpc

    torch.cuda.set_device(0)
    return mpc.lib()


def _p(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else None


def _quantise(lib, x, bits, mode, seed, noalloc):
    R, L = x.shape
    W = lib.mpc_quant_codes_words(R, L, bits) // R
    codes = torch.full((R, W), -1, dtype=torch.int32, device="cuda")
    scale = torch.full((R,), -1.0, device="cuda")
    minv = torch.full((R,), -1.0, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if noalloc:
        st = lib.mpc_quant_compress_noalloc(_p(x), R, L, bits, mode, seed, _p(codes), _p(scale),
                                            _p(minv), stream)
    else:
        nws = lib.mpc_quant_workspace_bytes(R, L, bits)
        ws = torch.empty(max(nws, 1), dtype=torch.uint8, device="cuda") if nws else None
        st = lib.mpc_quant_compress(_p(x), R, L, bits, mode, seed, _p(codes), _p(scale), _p(minv),
                                    _p(ws), nws, stream)
    assert st == 0, lib.mpc_last_error()
    assert lib.mpc_get_status(stream) == 0, lib.mpc_last_error()
    return codes.cpu().numpy().view(np.uint32), scale.cpu().numpy(), minv.cpu().numpy()


# Calls in a row: each has other rows and values than the one before, so anything an
# earlier call left in the shared scratch would show.  Rows longer than 65536 entries use
# the scratch (4-bit stochastic, and 6-bit codes that straddle words); 768-entry rows do
# not.
CALLS = [(96, 70001, 4, 1, (7 << 32) | 3, 0, 1.0), (300, 768, 8, 0, 0, 1, 1e-3),
         (40, 131075, 6, 0, 0, 2, 1e-2), (33, 65540, 6, 1, 5, 3, 1.0)]


def test_noalloc_matches_the_workspace_entry_point(lib):
    for R, L, bits, mode, seed, gen_seed, scale in CALLS:
        g = torch.Generator(device="cuda")
        g.manual_seed(gen_seed)
        x = torch.randn((R, L), generator=g, device="cuda") * scale
        want = _quantise(lib, x, bits, mode, seed, noalloc=False)
        got = _quantise(lib, x, bits, mode, seed, noalloc=True)
        for name, a, b in zip(("codes", "scale", "minv"), got, want):
            assert np.array_equal(a.view(np.uint32), b.view(np.uint32)), (R, L, bits, name)


def test_noalloc_at_the_row_limit(lib):
    """65536 rows of 65540 entries (the largest row count, every slot of the scratch in
    use), 2-bit codes, compared with the workspace entry point on the device."""
    R, L = 65536, 65540
    g = torch.Generator(device="cuda")
    g.manual_seed(4)
    x = torch.randn((R, L), generator=g, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    W = lib.mpc_quant_codes_words(R, L, 2) // R
    outs = []
    for noalloc in (False, True):
        codes = torch.full((R, W), -1, dtype=torch.int32, device="cuda")
        scale = torch.full((R,), -1.0, device="cuda")
        minv = torch.full((R,), -1.0, device="cuda")
        if noalloc:
            st = lib.mpc_quant_compress_noalloc(_p(x), R, L, 2, 0, 0, _p(codes), _p(scale),
                                                _p(minv), stream)
        else:
            nws = lib.mpc_quant_workspace_bytes(R, L, 2)
            ws = torch.empty(nws, dtype=torch.uint8, device="cuda")
            st = lib.mpc_quant_compress(_p(x), R, L, 2, 0, 0, _p(codes), _p(scale), _p(minv),
                                        _p(ws), nws, stream)
        assert st == 0, lib.mpc_last_error()
        assert lib.mpc_get_status(stream) == 0, lib.mpc_last_error()
        outs.append((codes, scale.view(torch.int32), minv.view(torch.int32)))
    del x
    for name, a, b in zip(("codes", "scale", "minv"), outs[1], outs[0]):
        assert torch.equal(a, b), name


def test_noalloc_rejects_too_many_rows(lib):
    p = ctypes.c_void_p(0x1000)
    st = lib.mpc_quant_compress_noalloc(p, 65537, 16, 4, 0, 0, p, p, p, None)
    assert st == 1
    assert b"static scratch" in lib.mpc_last_error()
