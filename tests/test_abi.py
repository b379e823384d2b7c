"""The C-ABI library loads on the CPU and exports every symbol its header declares, and
its host-side argument validation rejects bad calls before any launch (no GPU needed:
validation returns before any CUDA call)."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mpcomp.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mpc_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__ as g

    g.build()
    import paper_2401_07788_gb300 as mpc

    return mpc.lib()


def test_header_declares_the_boundary():
    names = declared_functions()
    for want in ("mpc_topk_compress", "mpc_topk_decompress", "mpc_ef_topk_compress",
                 "mpc_ef21_topk_compress", "mpc_aqsgd_compress", "mpc_aqsgd_decompress",
                 "mpc_quant_compress", "mpc_quant_decompress", "mpc_get_status",
                 "mpc_last_error", "mpc_topk_workspace_bytes", "mpc_quant_codes_words"):
        assert want in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_version(lib):
    assert lib.mpc_version() >= 100


def test_sizes(lib):
    # W = roundup4(ceil(L*b/32)) words per row
    assert lib.mpc_quant_codes_words(3, 768, 4) == 3 * 96
    assert lib.mpc_quant_codes_words(1, 31, 2) == 4
    assert lib.mpc_quant_codes_words(2, 16384, 8) == 2 * 4096
    assert lib.mpc_quant_codes_words(1, 5, 32) == 8
    assert lib.mpc_quant_codes_words(1, 5, 6) == 4  # 6-bit codes straddle words
    assert lib.mpc_quant_codes_words(1, 5, 17) == 0  # unsupported width
    assert lib.mpc_topk_workspace_bytes(128, 32768, 3276) == 0  # on-chip path
    assert lib.mpc_quant_workspace_bytes(128, 32768, 4) == 0
    # rows longer than 65536 go through the grid path in batches of up to 64 rows (about
    # 2^26 entries a batch), with a 256-byte-aligned workspace slice per row of a batch
    one = lib.mpc_topk_workspace_bytes(1, 70000, 7000)
    assert one > 0 and one % 256 == 0
    assert lib.mpc_topk_workspace_bytes(2, 70000, 7000) == 2 * one
    assert lib.mpc_topk_workspace_bytes(64, 70000, 7000) == 64 * one
    assert lib.mpc_topk_workspace_bytes(1000, 70000, 7000) == 64 * one
    big = lib.mpc_topk_workspace_bytes(1, 1 << 24, 1 << 20)
    assert lib.mpc_topk_workspace_bytes(16, 1 << 24, 1 << 20) == 4 * big
    whole = lib.mpc_topk_workspace_bytes(1, 1 << 30, 1 << 20)
    assert lib.mpc_topk_workspace_bytes(3, 1 << 30, 1 << 20) == whole


@pytest.mark.parametrize("args,code", [
    ((0x1000, 4, 16, 0), 1),        # k = 0
    ((0x1000, 4, 16, 17), 1),       # k > row_len
    ((0x1000, 4, 0, 1), 1),         # row_len = 0
    ((0x1000, -1, 16, 1), 1),       # rows < 0
    ((0, 4, 16, 2), 1),             # x NULL
    ((0x1002, 4, 16, 2), 1),        # x misaligned
])
def test_topk_validation(lib, args, code):
    x, rows, L, k = args
    st = lib.mpc_topk_compress(ctypes.c_void_p(x), rows, L, k, ctypes.c_void_p(0x2000),
                               ctypes.c_void_p(0x3000), None, 0, None)
    assert st == code
    assert lib.mpc_last_error()


def test_zero_rows_is_a_noop(lib):
    assert lib.mpc_topk_compress(None, 0, 16, 2, None, None, None, 0, None) == 0


def test_quant_validation(lib):
    p = ctypes.c_void_p(0x1000)
    for bad in (0, 17, 31, 33, -2):  # widths 1..16 and 32 only
        assert lib.mpc_quant_compress(p, 2, 16, bad, 0, 0, p, p, p, None, 0, None) == 1
        assert lib.mpc_quant_decompress(p, p, p, 2, 16, bad, p, None) == 1
        assert lib.mpc_quant_codes_words(2, 16, bad) == 0
    assert lib.mpc_quant_compress(p, 2, 16, 4, 7, 0, p, p, p, None, 0, None) == 1  # mode
    # W = roundup4(ceil(L * bits / 32)) words per row, for every width
    for bits in list(range(1, 17)) + [32]:
        for L in (1, 31, 100, 4097):
            w = -(-L * bits // 32)
            assert lib.mpc_quant_codes_words(3, L, bits) == 3 * (-(-w // 4) * 4)


def test_aqsgd_validation(lib):
    p = ctypes.c_void_p(0x1000)
    # sample_ids misaligned
    assert lib.mpc_aqsgd_compress(p, p, 10, ctypes.c_void_p(0x1004), 2, 3, 16, 2, p, p, None, 0,
                                  None) == 1
    assert lib.mpc_aqsgd_compress(p, p, 0, p, 2, 3, 16, 2, p, p, None, 0, None) == 1


def test_knobs(lib):
    assert lib.mpc_set_knob(99, 0) == 1
    assert lib.mpc_set_knob(2, 5) == 1
    assert lib.mpc_set_knob(2, 4) == 0  # rows of 1025..8192 entries without the band kernel
    assert lib.mpc_set_knob(2, 3) == 0  # rows of 8193..32768 entries on clusters only
    assert lib.mpc_set_knob(2, 0) == 0
    assert lib.mpc_set_knob(3, 2) == 1  # programmatic dependent launch: 0 or 1
    assert lib.mpc_set_knob(3, 0) == 0
    assert lib.mpc_set_knob(3, 1) == 0


def test_aqsgd_quant_validation(lib):
    p = ctypes.c_void_p(0x1000)
    q = ctypes.c_void_p(0x100000)

    def comp(num_samples=10, ids=p, n_ids=2, rps=3, L=16, bits=4, mode=0, ws=q, ws_bytes=1 << 20):
        return lib.mpc_aqsgd_quant_compress(p, p, num_samples, ids, n_ids, rps, L, bits, mode, 0,
                                            p, p, p, ws, ws_bytes, None)

    # the workspace holds d (rows x row_len fp32, rounded up to 256 bytes), plus the
    # quantiser's own for rows longer than its on-chip path
    assert lib.mpc_aqsgd_quant_workspace_bytes(2, 3, 16, 4) == 512  # 6 x 16 x 4 = 384 -> 512
    assert lib.mpc_aqsgd_quant_workspace_bytes(4, 2, 256, 4) == 8 * 256 * 4
    assert lib.mpc_aqsgd_quant_workspace_bytes(1, 1, 100000, 4) == 400128 + 8
    assert lib.mpc_aqsgd_quant_workspace_bytes(2, 3, 16, 17) == 0
    assert lib.mpc_aqsgd_quant_workspace_bytes(0, 3, 16, 4) == 0
    assert comp(bits=17) == 1 and comp(bits=0) == 1
    assert comp(mode=7) == 1
    assert comp(num_samples=0) == 1 and comp(rps=0) == 1 and comp(n_ids=-1) == 1
    assert comp(ids=ctypes.c_void_p(0x1004)) == 1       # sample ids misaligned
    assert comp(ws=None) == 3 and comp(ws_bytes=255) == 3  # workspace missing or short
    assert comp(n_ids=0, ws=None, ws_bytes=0) == 0      # nothing to do
    dec = lambda **kw: lib.mpc_aqsgd_quant_decompress(  # noqa: E731
        p, p, p, p, kw.get("num_samples", 10), kw.get("ids", p), kw.get("n_ids", 2), 3, 16,
        kw.get("bits", 4), None)
    assert dec(bits=33) == 1 and dec(num_samples=0) == 1
    assert dec(ids=ctypes.c_void_p(0x1002)) == 1
    assert dec(n_ids=0) == 0


def test_gather_and_efmix_validation(lib):
    p = ctypes.c_void_p(0x1000)
    # index reuse: the payload shape rules of TopK
    assert lib.mpc_topk_gather(p, 2, 16, p, 0, p, None) == 1      # k = 0
    assert lib.mpc_topk_gather(p, 2, 16, p, 17, p, None) == 1     # k > row_len
    assert lib.mpc_topk_gather(None, 2, 16, p, 4, p, None) == 1   # g NULL
    assert lib.mpc_topk_gather(p, 0, 16, p, 4, p, None) == 0      # no rows
    # EF-mixed: the two shares' index and saved-value arrays (256-byte rounded) come first
    k = 7
    share = -(-(3 * ((k + 1) // 2) * 4) // 256) * 256
    assert lib.mpc_efmix_workspace_bytes(3, 64, k) >= 2 * share
    assert lib.mpc_efmix_workspace_bytes(3, 64, 0) == 0
    need = lib.mpc_efmix_workspace_bytes(3, 64, k)
    ws = ctypes.c_void_p(0x100000)
    call = lambda ws, n: lib.mpc_efmix_topk_compress(p, p, 3, 64, k, p, p, ws, n, None)  # noqa: E731
    assert call(None, 0) == 3                       # workspace missing
    assert call(ws, need - 1) == 3                  # workspace short
    assert call(ctypes.c_void_p(0x100010), need) == 1  # workspace not 256-byte aligned
