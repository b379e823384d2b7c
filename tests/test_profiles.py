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
    lines = open(os.path.join(ROOT, "profiles", "dram_traffic.txt")).read().splitlines()
    digests = [ln.split()[1] for ln in lines if ln.startswith("source_digest ")]
    assert len(digests) == 1 and len(digests[0]) == 16
    entries = {ln.split()[0]: float(ln.split()[1]) for ln in lines
               if ln.strip() and not ln.startswith("#") and not ln.startswith("source_digest")}
    b = _bench()
    kern = lambda o: ("topk_cta_kernel" if "topk_compress" in o else  # noqa: E731
                      "topk_decompress_rows_kernel" if "decompress K" in o else
                      "quant_cta_kernel" if "quant_compress" in o else "dequant_rows_kernel")
    ops = ["ef_topk_compress K=%d%%" % p for p in b.TOPK_PCTS]
    ops += ["topk_decompress K=%d%%" % p for p in b.TOPK_PCTS]
    for bits in b.BITS:
        for sr in ("nearest", "stochastic"):
            ops += ["quant_compress %d-bit %s" % (bits, sr), "quant_decompress %d-bit %s" % (bits, sr)]
    for o in ops:
        key = kern(o) + ":" + o.replace(" ", "_")
        assert key in entries and entries[key] > 0, key
    # inputs read once: an error-feedback TopK launch reads x and err, 2 x 16.8 MB
    ef = entries["topk_cta_kernel:ef_topk_compress_K=5%"]
    assert 2 * 4 * b.R * b.L * 0.99 <= ef <= 2 * 4 * b.R * b.L * 1.05


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
