"""The committed ncu traffic table that bench.py reads for roofline.traffic: it parses,
names a source digest, and holds a per-launch DRAM figure for every operator of the
benchmark step (no GPU needed)."""

import importlib.util
import os

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_traffic_table_parses():
    """The table parses, names one source digest, and every entry is a call of the
    headline step with a positive byte count, not below the bytes the call must read."""
    lines = open(os.path.join(ROOT, "profiles", "dram_traffic.txt")).read().splitlines()
    digests = [ln.split()[1] for ln in lines if ln.startswith("source_digest ")]
    assert len(digests) == 1 and len(digests[0]) == 16
    entries = {}
    for ln in lines:
        if ln.strip() and not ln.startswith("#") and not ln.startswith("source_digest"):
            name, value = ln.rsplit(None, 1)
            entries[name] = float(value)
    b = _bench()
    names = set(b.headline_call_names())
    assert entries, "empty traffic table"
    N = 1 << b.LOG2N
    for name, v in entries.items():
        assert name in names, name
        # every compress call reads its 4 GiB input at least once
        if "compress" in name and "decompress" not in name:
            assert v >= 4 * N * 0.99, (name, v)


def test_headline_calls():
    """36 compress+decompress pairs per headline step: for each of the four row lengths,
    TopK and EF-TopK at three K and three code widths."""
    b = _bench()
    names = b.headline_call_names()
    assert len(names) == 72 and len(set(names)) == 72
    assert sum("decompress" in n for n in names) == 36
    for L in ("768", "4096", "65536", "N"):
        assert sum(("L=%s " % L) in n for n in names) == 18


def test_step_branch_layouts():
    """Every concurrent-branch layout of the benchmark step puts each of its nine pairs on
    a branch that exists, keeps a pair's two launches together (one branch per pair) and
    uses every branch; one branch is the launches in order."""
    b = _bench()
    for nb, f in b.BRANCH_OF.items():
        got = []
        for i in range(9):
            sr = None if i < 3 else bool((i - 3) % 2)
            br = f(i, sr)
            assert 0 <= br < nb, (nb, i, br)
            got.append(br)
        assert sorted(set(got)) == list(range(nb)), (nb, got)
        assert nb in b.BRANCH_TEXT
    assert set(b.BRANCH_OF[1](i, None if i < 3 else False) for i in range(9)) == {0}


def test_algorithmic_bytes():
    """Minimum HBM bytes per call: TopK 4N + 8kR, error feedback / EF21 / AQ-SGD
    12N + 8kR, decompression 8kR + 4N, (de)quantisation 4N + ceil(N b / 8) + 8R."""
    b = _bench()
    R, L, k = 2, 10, 3
    assert b.algorithmic_bytes(R, L, k=k, op="topk") == 4 * 20 + 8 * 3 * 2
    assert b.algorithmic_bytes(R, L, k=k, op="ef_topk") == 12 * 20 + 8 * 3 * 2
    assert b.algorithmic_bytes(R, L, k=k, op="delta_topk") == 12 * 20 + 8 * 3 * 2
    assert b.algorithmic_bytes(R, L, k=k, op="topk_decompress") == 8 * 3 * 2 + 4 * 20
    assert b.algorithmic_bytes(R, L, bits=3, op="quant") == 4 * 20 + 8 + 8 * 2  # 60 bits -> 8 B
    assert b.algorithmic_bytes(R, L, bits=4, op="dequant") == 4 * 20 + 10 + 8 * 2
    # the headline at 2^30: a whole-tensor error-feedback TopK at K = 50 % is 17.2 GB
    N = 1 << 30
    assert b.algorithmic_bytes(1, N, k=N // 2, op="ef_topk") == 12 * N + 4 * N


def test_kernels_of_name_library_kernels():
    """Every kernel bench.py attributes a headline call's launches to is a __global__
    function of the library's sources (the traffic table and the launch list map ncu's
    launches to calls through these lists)."""
    import re

    b = _bench()
    csrc = os.path.join(ROOT, "paper_2401_07788_gb300", "csrc")
    text = "".join(open(os.path.join(csrc, f)).read() for f in os.listdir(csrc)
                   if f.endswith((".cu", ".cuh")))
    bounds = r"__launch_bounds__\((?:[^()]|\([^()]*\))*\)\s*"  # one level of nesting
    globals_ = set(re.findall(r"__global__\s+void\s+(?:%s)?(\w+)\s*\(" % bounds, text))
    N = 1 << b.LOG2N
    for op in ("topk", "ef_topk", "topk_decompress", "quant", "dequant"):
        for L in (768, 4096, 65536, N):
            ks = b.kernels_of(op, L)
            assert ks, (op, L)
            for kname in ks:
                assert kname in globals_, (op, L, kname)
    # a whole-tensor TopK is one batch of 23 launches, a whole-tensor quantisation 3
    assert len(b.kernels_of("topk", N)) == 23
    assert len(b.kernels_of("quant", N)) == 3
