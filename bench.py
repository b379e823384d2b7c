#!/usr/bin/env python3
"""Benchmark of libmpcomp: compress+decompress GB/s (input bytes) and the fraction of HBM
bandwidth per operator, on one GB300.

Workload (the CNN stage boundary, [128,128,16,16] fp32 = 128 rows x 32768): one step is
one boundary crossing of every operator the workload sweeps, on that step's tensors:
  forward : error-feedback TopK at K = 5, 10, 30 % (one error buffer per K, carried
            across steps) of the activation ReLU(N(0,1)) drifting by 0.1*N(0,1) per step,
            each followed by TopK decompression;
  backward: 2/4/8-bit min-max quantisation of the gradient N(0, sigma=1e-3), round to
            nearest and stochastic (seed (seed << 32) | step), each followed by
            dequantisation.
value = sum over the 9 compress+decompress pairs of the input bytes (4 x 128 x 32768) /
device time of the step.  Each step is one CUDA graph of the 18 library launches (one
graph per slot of a pool of 4 pre-drawn steps, so inputs differ from step to step), with
no event nodes inside; the nine pairs are independent and run as concurrent branches of
the graph (--branches).  L2 is flushed before every timed step by writing and then
reading a 256 MiB buffer (so the step's inputs are cold and the flush leaves no dirty
lines for the first launch to write back), outside the timed interval.  Per-launch
shares come from a second timed pass whose graphs run the 18 launches in order and
record an event after every launch; the dominant launch's duration (for `roofline`)
from 200 launches of it in a row between two events on its stream, the inputs cycling
through 8 copies (twice the L2) so that each launch reads cold inputs, and, for
reference, from single launches between two events (which adds ~5 us to any launch).  `e2e` runs
the steps through the Python API with the step's inputs copied from pinned host memory
and two outputs copied back inside the timed region.  `operators` times every operator
of the path on its own workload: a CUDA graph of 8 x (L2 flush, launch) against a graph
of the 8 flushes alone, the difference divided by 8.

`--impl reference` times the CPU oracle (single-threaded C) on a bounded sample of the
same step: 16 of the 128 rows.
"""

from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

METRIC = "compress+decompress GB/s (input bytes) and % of HBM roofline per operator at 1 GB300"
UNIT = "GB/s"
WORKLOAD = "CNN stage boundary [128,128,16,16] fp32"
R, L = 128, 32768
TOPK_PCTS = (5, 10, 30)
BITS = (2, 4, 8)
POOL = 4
SAMPLE_ROWS = 16


def parse_args():
    p = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=1000)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=("ours", "reference"), default="ours")
    p.add_argument("--no-operators", action="store_true", help="skip the per-operator table")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--sweep", action="store_true",
                   help="only the size sweep: N = 2^20..2^30 entries, L in {768, 4096, 65536, N}; "
                        "prints one JSON line with the table (not the benchmark line)")
    p.add_argument("--branches", type=int, default=6, choices=(1, 2, 3, 5, 6, 9),
                   help="concurrent streams inside the step graph (1 = all launches in order)")
    return p.parse_args()


# ---------------------------------------------------------------------------------------
# process group (one process per GPU; independent replicas, no data exchange)
# ---------------------------------------------------------------------------------------

def dist_env():
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0")),
            int(os.environ.get("WORLD_SIZE", "1")))


def init_dist(world: int, backend: str):
    if world > 1:
        import torch.distributed as dist

        if not dist.is_initialized():
            dist.init_process_group(backend=backend)


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


def aggregate(units: float, seconds: float, world: int, device) -> tuple[float, float]:
    """Whole-job units (sum over ranks) and time (max over ranks)."""
    if world == 1:
        return units, seconds
    import torch.distributed as dist

    t = torch.tensor([units, seconds], dtype=torch.float64, device=device)
    u = t[:1].clone()
    s = t[1:].clone()
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    dist.all_reduce(s, op=dist.ReduceOp.MAX)
    return float(u.item()), float(s.item())


# ---------------------------------------------------------------------------------------
# peaks, clocks, traffic records
# ---------------------------------------------------------------------------------------

def hbm_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


def source_digest() -> str:
    import hashlib

    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2401_07788_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str):
    """DRAM bytes per launch from the committed ncu summary, if taken on this source."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    try:
        lines = open(path).read().splitlines()
    except OSError:
        return None
    digest = None
    table = {}
    for ln in lines:
        parts = ln.split()
        if len(parts) >= 2 and parts[0] == "source_digest":
            digest = parts[1]
        elif len(parts) >= 2 and not ln.startswith("#"):
            try:
                table[parts[0]] = float(parts[1])
            except ValueError:
                pass
    if digest != source_digest():
        return None
    return table.get(kernel)


class ClockSampler:
    """SM clock and clock-event reasons sampled every ~2 ms while the benchmark runs,
    through NVML (read-only queries), else through nvidia-smi."""

    # NVML clock-event reason bits
    REASONS = ((0x4, "sw_power_cap"), (0x8, "hw_slowdown"), (0x20, "sw_thermal_slowdown"),
               (0x40, "hw_thermal_slowdown"), (0x80, "hw_power_brake_slowdown"))

    def __init__(self, device_index: int, interval_s: float = 0.002):
        self.interval = interval_s
        self.samples = []  # (sm_mhz, reason bits)
        self.max_mhz = None
        self.source = None
        self.bus = None
        try:
            p = torch.cuda.get_device_properties(device_index)
            self.bus = "%08X:%02X:%02X.0" % (p.pci_domain_id, p.pci_bus_id, p.pci_device_id)
        except Exception:
            pass
        self.nvml = self._open_nvml()

    def _open_nvml(self):
        import ctypes

        try:
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0 or self.bus is None:
                return None
            h = ctypes.c_void_p()
            if lib.nvmlDeviceGetHandleByPciBusId_v2(self.bus.encode(), ctypes.byref(h)) != 0:
                return None
            reasons = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                lib.nvmlDeviceGetCurrentClocksThrottleReasons
            mx = ctypes.c_uint()
            if lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:
                self.max_mhz = float(mx.value)
            return (lib, h, reasons)
        except (OSError, AttributeError):
            return None

    def _sample_nvml(self):
        import ctypes

        lib, h, reasons = self.nvml
        mhz, bits = ctypes.c_uint(), ctypes.c_ulonglong()
        if lib.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(mhz)) == 0 and \
                reasons(h, ctypes.byref(bits)) == 0:
            self.samples.append((float(mhz.value), int(bits.value)))

    def __enter__(self):
        import threading

        self.stop = threading.Event()
        self.proc = None
        if self.nvml is not None:
            self.source = "nvml"
            self._sample_nvml()

            def loop():
                while not self.stop.wait(self.interval):
                    self._sample_nvml()

            self.thread = threading.Thread(target=loop, daemon=True)
            self.thread.start()
        else:
            self.thread = None
            self.out = os.path.join("/tmp", "mpc_clocks_%d.csv" % os.getpid())
            cmd = ["nvidia-smi", "--query-gpu=clocks.sm,clocks.max.sm,"
                   "clocks_event_reasons.active", "--format=csv,noheader,nounits", "-lms", "20"]
            if self.bus:
                cmd += ["-i", self.bus]
            try:
                self.fh = open(self.out, "w")
                self.proc = subprocess.Popen(cmd, stdout=self.fh, stderr=subprocess.DEVNULL)
                self.source = "nvidia-smi"
                time.sleep(0.5)  # let it start before the timed region
            except OSError:
                self.proc = None
        return self

    def __exit__(self, *exc):
        self.stop.set()
        if self.thread is not None:
            self.thread.join()
            self._sample_nvml()
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.fh.close()
            try:
                for row in open(self.out).read().splitlines():
                    f = [c.strip() for c in row.split(",")]
                    try:
                        self.samples.append((float(f[0]), int(f[2], 16)))
                        self.max_mhz = float(f[1])
                    except (ValueError, IndexError):
                        continue
                os.remove(self.out)
            except OSError:
                pass

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": [],
                    "samples": 0, "source": self.source or "unavailable"}
        reasons = sorted({name for _, b in self.samples for bit, name in self.REASONS if b & bit})
        return {"sm_mhz": statistics.median(s for s, _ in self.samples),
                "sm_max_mhz": self.max_mhz, "reasons": reasons,
                "samples": len(self.samples), "source": self.source}


# ---------------------------------------------------------------------------------------
# the workload
# ---------------------------------------------------------------------------------------

def algorithmic_bytes(R_, L_, k=None, bits=None, op=""):
    """Minimum HBM bytes of one launch: inputs and buffers read once, payload and buffers
    written once."""
    N = R_ * L_
    if op == "ef_topk":
        return 12 * N + 8 * k * R_
    if op == "topk":
        return 4 * N + 8 * k * R_
    if op == "topk_decompress":
        return 8 * k * R_ + 4 * N
    if op == "delta_topk":  # EF21 / AQ-SGD: state written only where kept
        return 8 * N + 12 * k * R_
    if op == "efmix_topk":  # x and err read, err written, payload written
        return 12 * N + 8 * k * R_
    if op == "topk_gather":  # indices read, values gathered, payload written
        return 12 * k * R_
    if op == "aqsgd_decompress":
        return 8 * k * R_ + 8 * k * R_
    if op == "aqsgd_quant":  # x and buffer rows read, buffer rows and codes written
        return 12 * N + (N * bits + 7) // 8 + 8 * R_
    if op == "aqsgd_dequant_add":  # codes and buffer rows read, buffer rows written
        return 8 * N + (N * bits + 7) // 8 + 8 * R_
    if op in ("quant", "dequant"):
        return 4 * N + (N * bits + 7) // 8 + 8 * R_
    raise ValueError(op)


class Step:
    """Pre-allocated tensors and the launch sequence of one boundary step."""

    def __init__(self, mpc, synth, device, seed: int):
        self.mpc = mpc
        gen = synth.generator(seed, device)
        x = synth.relu_normal((R, L), seed, device, gen=gen)
        self.xs, self.gs = [], []
        for t in range(POOL):
            self.xs.append(x)
            self.gs.append(synth.normal((R, L), 1000 + 100 * seed + t, device, std=1e-3))
            x = synth.drift(x, 0.1, gen)
        self.ks = {p: synth.k_of(L, p) for p in TOPK_PCTS}
        self.errs = {p: torch.zeros((R, L), device=device) for p in TOPK_PCTS}
        self.vals = {p: torch.empty((R, self.ks[p]), device=device) for p in TOPK_PCTS}
        self.idx = {p: torch.empty((R, self.ks[p]), dtype=torch.int32, device=device)
                    for p in TOPK_PCTS}
        # every pair has its own outputs, so that pairs on different streams share nothing
        QS = [(b, sr) for b in BITS for sr in (False, True)]
        self.y = {p: torch.empty((R, L), device=device) for p in TOPK_PCTS}
        self.gy = {q: torch.empty((R, L), device=device) for q in QS}
        W = {b: mpc.mpc_quant_codes_words(R, L, b) // R for b in BITS}
        self.codes = {q: torch.empty((R, W[q[0]]), dtype=torch.int32, device=device) for q in QS}
        self.scale = {q: torch.empty(R, device=device) for q in QS}
        self.minv = {q: torch.empty(R, device=device) for q in QS}
        self.seed = seed
        self.ops = []  # (name, bytes) in launch order
        for p in TOPK_PCTS:
            self.ops.append(("ef_topk_compress K=%d%%" % p,
                             algorithmic_bytes(R, L, k=self.ks[p], op="ef_topk")))
            self.ops.append(("topk_decompress K=%d%%" % p,
                             algorithmic_bytes(R, L, k=self.ks[p], op="topk_decompress")))
        for b in BITS:
            for sr in (False, True):
                tag = "%d-bit %s" % (b, "stochastic" if sr else "nearest")
                self.ops.append(("quant_compress " + tag, algorithmic_bytes(R, L, bits=b, op="quant")))
                self.ops.append(("quant_decompress " + tag, algorithmic_bytes(R, L, bits=b, op="dequant")))
        self.input_bytes = 9 * 4 * R * L  # 9 compress+decompress pairs

    def rotation(self, i: int, n_sets: int, step: int = 0):
        """Launch i of the step over n_sets independent copies of the inputs it reads and
        the dense outputs it writes (payloads and codes are shared): one callable per
        set, for back-to-back timing on inputs that L2 no longer holds."""
        m = self.mpc
        name = self.ops[i][0]
        fns = []
        for s_ in range(n_sets):
            if name.startswith("ef_topk_compress"):
                p = int(name.split("K=")[1].rstrip("%"))
                x = self.xs[s_ % POOL].clone()
                e = self.errs[p].clone()
                fns.append(lambda x=x, e=e, p=p: m.mpc_ef_topk_compress(
                    x, e, self.ks[p], self.vals[p], self.idx[p]))
            elif name.startswith("topk_decompress"):
                p = int(name.split("K=")[1].rstrip("%"))
                y = torch.empty_like(self.y[p])
                fns.append(lambda y=y, p=p: m.mpc_topk_decompress(self.vals[p], self.idx[p], L, y=y))
            else:
                b_ = int(name.split()[1].split("-")[0])
                q = (b_, name.endswith("stochastic"))
                if name.startswith("quant_compress"):
                    g = self.gs[s_ % POOL].clone()
                    fns.append(lambda g=g, q=q: m.mpc_quant_compress(
                        g, q[0], stochastic=q[1], seed=(self.seed << 32) | step,
                        codes=self.codes[q], scale=self.scale[q], minv=self.minv[q]))
                else:
                    y = torch.empty_like(self.gy[q])
                    fns.append(lambda y=y, q=q: m.mpc_quant_decompress(
                        self.codes[q], self.scale[q], self.minv[q], L, q[0], y=y))
        return fns

    def launch(self, slot: int, step: int, events=None, x=None, g=None, side=None,
               y=None, gy=None, only=None):
        """Enqueue the step's 18 launches.  events: one event recorded after each launch;
        only: enqueue launch `only` alone (timing of one launch on its own).
        side: streams for concurrent branches (the nine pairs are independent; BRANCH_OF
        maps a pair to its branch, branch 0 being the current stream).  The branches fork
        from and join back into the current stream.  y, gy: outputs to use instead of the
        step's own, by TopK percent and by (bits, stochastic)."""
        m = self.mpc
        x = self.xs[slot] if x is None else x
        g = self.gs[slot] if g is None else g
        e = iter(events) if events is not None else None
        n = [0]

        def op(fn):
            fn()
            if e is not None:
                next(e).record()
            n[0] += 1

        ys = {**self.y, **(y or {})}
        gys = {**self.gy, **(gy or {})}
        nb = 1 + len(side or [])
        seq = []  # (branch, launch) in the order of self.ops
        for i, p in enumerate(TOPK_PCTS):
            br = BRANCH_OF[nb](i, None)
            seq.append((br, lambda p=p: m.mpc_ef_topk_compress(x, self.errs[p], self.ks[p],
                                                               self.vals[p], self.idx[p])))
            seq.append((br, lambda p=p: m.mpc_topk_decompress(self.vals[p], self.idx[p], L,
                                                              y=ys[p])))
        for b in BITS:
            for sr in (False, True):
                q = (b, sr)
                br = BRANCH_OF[nb](len(seq) // 2, sr)
                seq.append((br, lambda q=q: m.mpc_quant_compress(
                    g, q[0], stochastic=q[1], seed=(self.seed << 32) | step, codes=self.codes[q],
                    scale=self.scale[q], minv=self.minv[q])))
                seq.append((br, lambda q=q: m.mpc_quant_decompress(
                    self.codes[q], self.scale[q], self.minv[q], L, q[0], y=gys[q])))
        if only is not None:
            seq[only][1]()
            return
        if not side:
            for _, fn in seq:
                op(fn)
            return
        main = torch.cuda.current_stream()
        streams = [main] + list(side)
        fork = torch.cuda.Event()
        fork.record(main)
        for s in side:
            s.wait_event(fork)
        for br, fn in seq:
            with torch.cuda.stream(streams[br]):
                fn()
        for s in side:
            main.wait_stream(s)


# Branch of pair i (0-2 the TopK pairs, 3-8 the quantisation pairs; sr = stochastic
# rounding) for a step of n concurrent branches.
BRANCH_OF = {
    1: lambda i, sr: 0,
    2: lambda i, sr: 0 if i < 3 else 1,
    3: lambda i, sr: 0 if i < 3 else 1 + int(sr),
    5: lambda i, sr: i if i < 3 else 3 + int(sr),
    6: lambda i, sr: i if i < 3 else 3 + (i - 3) // 2,
    9: lambda i, sr: i,
}

BRANCH_TEXT = {
    1: "the 18 launches in order on one stream",
    2: "two concurrent branches (the three TopK pairs; the six quantisation pairs), each in "
       "order, forked from and joined into one stream",
    3: "three concurrent branches (the three TopK pairs; the nearest quantisation pairs; the "
       "stochastic ones), each in order, forked from and joined into one stream",
    5: "five concurrent branches (each TopK pair; the nearest quantisation pairs; the "
       "stochastic ones), each in order, forked from and joined into one stream",
    6: "six concurrent branches (each TopK pair; the 2-, 4- and 8-bit quantisation pairs), "
       "each in order, forked from and joined into one stream",
    9: "nine concurrent branches (one per compress+decompress pair), forked from and joined "
       "into one stream",
}


def make_event(external: bool):
    if external:
        try:
            return torch.cuda.Event(enable_timing=True, external=True)
        except TypeError:
            return None
    return torch.cuda.Event(enable_timing=True)


def run_ours(args, rank, local, world):
    import paper_2401_07788_gb300 as mpc
    from paper_2401_07788_gb300 import synth

    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    init_dist(world, "nccl")
    mpc.lib()
    seed = rank % 10
    st = Step(mpc, synth, device, seed)
    n_ops = len(st.ops)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=device)
    flush_sink = torch.empty((), dtype=torch.int64, device=device)
    stream = torch.cuda.Stream(device)
    side = [torch.cuda.Stream(device) for _ in range(args.branches - 1)]
    torch.cuda.synchronize()

    def flush_l2(i):
        # write then read a buffer twice the size of L2: the step's inputs leave
        # L2, and the flush leaves no dirty lines whose write-back the first
        # launch of the step would pay for
        flush.fill_(i & 0xff)
        torch.sum(flush.view(torch.int64), dim=0, out=flush_sink)

    # eager warm-up (sets kernel attributes) before capture
    with torch.cuda.stream(stream):
        for w in range(2):
            st.launch(w % POOL, w)
            st.launch(w % POOL, w, side=side)
    stream.synchronize()
    assert mpc.mpc_get_status(stream) == 0, mpc.mpc_last_error()

    # One graph per pool slot.  Event nodes inside a graph cost ~5 us each, so the
    # headline steps replay event-free graphs; per-launch times come from a second
    # timed pass with an event after every launch (shares of the step), and the
    # dominant launch's duration from launches of it in a row on cold inputs
    # (time_back_to_back).
    if make_event(external=True) is None:
        raise RuntimeError("torch.cuda.Event(external=True) is required")
    keep = []  # events referenced by graph nodes must outlive the graphs

    def capture(slot, **kw):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            st.launch(slot, slot, **kw)
        return g

    plain = [capture(slot, side=side) for slot in range(POOL)]
    evsets = [[make_event(True) for _ in range(n_ops)] for _ in range(POOL)]
    keep.append(evsets)
    evented = [capture(slot, events=evsets[slot]) for slot in range(POOL)]
    torch.cuda.synchronize()

    def timed_pass(graphs, after_step=None, sampler=None):
        starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        with torch.cuda.stream(stream):
            for w in range(args.warmup):
                flush_l2(w)
                graphs[w % POOL].replay()
        stream.synchronize()
        barrier(world)
        torch.cuda.synchronize()
        if sampler is not None:
            sampler.__enter__()
        t0 = time.perf_counter()
        with torch.cuda.stream(stream):
            for i in range(args.steps):
                flush_l2(i)
                starts[i].record(stream)
                graphs[i % POOL].replay()
                ends[i].record(stream)
                if after_step is not None and ((i + 1) % POOL == 0 or i == args.steps - 1):
                    # events inside a graph belong to its slot: read them before reuse
                    stream.synchronize()
                    for j in range(i - (i % POOL), i + 1):
                        after_step(j, starts[j], ends[j])
        stream.synchronize()
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
        if sampler is not None:
            sampler.__exit__(None, None, None)
        barrier(world)
        return sum(starts[i].elapsed_time(ends[i]) for i in range(args.steps)) / 1e3, wall

    for p in TOPK_PCTS:
        st.errs[p].zero_()
    sampler = ClockSampler(local)
    dev_s, wall = timed_pass(plain, sampler=sampler)
    clocks = sampler.summary()

    op_ms = [0.0] * n_ops

    def read_ops(j, start, end):
        prev = start
        for i, ev in enumerate(evsets[j % POOL]):
            op_ms[i] += prev.elapsed_time(ev)
            prev = ev

    timed_pass(evented, read_ops)
    dom = max(range(n_ops), key=lambda j: op_ms[j])
    dom_ms = time_back_to_back(st, dom, stream, flush_l2)
    alone_ms = time_alone(st, dom, stream, flush_l2, min(args.steps, 300), args.warmup)
    status = mpc.mpc_get_status(stream)
    if status != 0:
        raise RuntimeError("device status %d: %s" % (status, mpc.mpc_last_error()))

    units, secs = aggregate(st.input_bytes * args.steps, dev_s, world, device)
    value = units / secs / 1e9

    # roofline of the dominant kernel (largest share of the step)
    peak, peak_kind = hbm_peak()
    name, nbytes = st.ops[dom]
    avg_ms = dom_ms
    achieved = nbytes / (avg_ms / 1e3) / 1e9
    kern = "topk_cta_kernel" if "topk_compress" in name else (
        "topk_decompress_rows_kernel" if "decompress K" in name else (
            "quant_cta_kernel" if "quant_compress" in name else "dequant_rows_kernel"))
    traffic = recorded_traffic(kern + ":" + name.replace(" ", "_"))
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "traffic": traffic,
                "kernel": kern, "op": name, "algorithmic_bytes": nbytes,
                "avg_launch_us": round(avg_ms * 1e3, 2),
                "share_of_step": round(op_ms[dom] / max(sum(op_ms), 1e-9), 4),
                "peak_source": peak_kind,
                "timing": "200 launches in a row on its stream between two CUDA events, "
                          "inputs cycling through 8 copies (twice the L2), so every launch "
                          "reads cold inputs",
                "alone_us": round(alone_ms * 1e3, 2),
                "alone_timing": "one launch after an L2 flush between two events behind a "
                                "GPU-side sleep (median of %d); includes the ~5 us an event "
                                "pair adds around any launch" % min(args.steps, 300)}
    per_op = {st.ops[j][0]: {"avg_us": round(op_ms[j] / args.steps * 1e3, 2),
                             "GBps": round(st.ops[j][1] / (op_ms[j] / args.steps / 1e3) / 1e9, 1)}
              for j in range(n_ops)}

    # end to end through the Python API: host inputs in, two outputs back, no graphs
    e2e = run_e2e(args, st, stream, side, world, device)

    operators = None
    if not args.no_operators and rank == 0:
        operators = measure_operators(mpc, synth, device, stream, peak)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(budget_s=10.0)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(secs * 1e3 / args.steps, 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": WORKLOAD, "rows": R, "row_len": L,
                       "topk_percents": list(TOPK_PCTS), "bits": list(BITS),
                       "rounding": ["nearest", "stochastic"], "launches_per_step": n_ops,
                       "step": "one CUDA graph per step (no event nodes inside); " + BRANCH_TEXT[args.branches],
                       "l2": "256 MiB buffer "
                       "written then read before each timed step, outside the timed interval "
                       "(inputs cold, no dirty lines left by the flush)", "parallelism":
                       "replicas" if world > 1 else "single GPU"},
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": n_ops * args.steps, "clocks": clocks,
            "wall_s": round(wall, 3), "per_op": per_op,
            "per_op_timing": "an event after every launch inside a graph of the 18 launches in "
                             "order on one stream (second pass; each interval includes the ~5 us "
                             "of an event node)",
            "operators": operators,
        }
        print(json.dumps(line), flush=True)


def time_back_to_back(st, i, stream, flush_l2, rounds=25, n_sets=8):
    """Average device time (ms) of launch i of the step over rounds x n_sets launches in
    a row on one stream, between two CUDA events: the launches cycle through n_sets
    copies of their inputs (8 x 33.5 MB for an error-feedback TopK, twice the L2), so
    each one reads inputs that L2 no longer holds, and the ~5 us that an event pair adds
    around any single launch is spread over all of them.  One round is captured as a
    CUDA graph so that the host's enqueue never paces the device."""
    fns = st.rotation(i, n_sets)
    with torch.cuda.stream(stream):
        for fn in fns:
            fn()
        stream.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for fn in fns:
                fn()
        g.replay()
        flush_l2(0)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(rounds):
            g.replay()
        b.record(stream)
        stream.synchronize()
    return a.elapsed_time(b) / (rounds * n_sets)


def time_alone(st, i, stream, flush_l2, n, warmup):
    """Median device time (ms) of launch i of the step on its own, on cold inputs: after
    each L2 flush a GPU-side sleep of ~50 us lets the host enqueue the two events and
    the launch before the stream reaches them, so the interval holds the launch alone."""
    with torch.cuda.stream(stream):
        for w in range(warmup):
            flush_l2(w)
            st.launch(w % POOL, w, only=i)
        stream.synchronize()
        pairs = []
        for s in range(n):
            flush_l2(s)
            torch.cuda._sleep(100_000)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            st.launch(s % POOL, s, only=i)
            b.record(stream)
            pairs.append((a, b))
        stream.synchronize()
    ts = [a.elapsed_time(b) for a, b in pairs]
    return statistics.median(ts)


def run_e2e(args, st, stream, side, world, device):
    """The step end to end through the Python API: every step copies its two inputs from
    pinned host memory to the device and two of its results back, inside the timed
    region.  Copies and compute are pipelined over two slots (inputs and read-back
    outputs double-buffered; step s+1's inputs go up while step s computes and step
    s-1's results come down), each copy on its own stream; the compute of a slot is the
    step's API calls captured once into a CUDA graph (its branches as in the headline)."""
    mpc = st.mpc
    hx = [t.cpu().pin_memory() for t in st.xs]
    hg = [t.cpu().pin_memory() for t in st.gs]
    k10, q8 = 10, (8, True)  # read back: the K=10% activation, the 8-bit stochastic gradient
    dx = [torch.empty_like(st.xs[0]) for _ in range(2)]
    dg = [torch.empty_like(st.gs[0]) for _ in range(2)]
    dy = [torch.empty((R, L), device=device) for _ in range(2)]
    dgy = [torch.empty((R, L), device=device) for _ in range(2)]
    hy = [torch.empty((R, L), pin_memory=True) for _ in range(2)]
    hgy = [torch.empty((R, L), pin_memory=True) for _ in range(2)]
    up = [torch.cuda.Stream(device) for _ in range(2)]
    down = [torch.cuda.Stream(device) for _ in range(2)]
    ev = lambda: [torch.cuda.Event() for _ in range(2)]  # noqa: E731
    x_in, g_in, done, y_out, g_out = ev(), ev(), ev(), ev(), ev()

    graphs = []
    for slot in range(2):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            st.launch(slot, slot, x=dx[slot], g=dg[slot], side=side,
                      y={k10: dy[slot]}, gy={q8: dgy[slot]})
        graphs.append(g)

    def one(s):
        b = s % 2
        for stm, dst, src, e in ((up[0], dx[b], hx[s % POOL], x_in[b]),
                                 (up[1], dg[b], hg[s % POOL], g_in[b])):
            stm.wait_event(done[b])  # the slot's previous compute has read it
            with torch.cuda.stream(stm):
                dst.copy_(src, non_blocking=True)
                e.record(stm)
        for e in (x_in[b], g_in[b], y_out[b], g_out[b]):
            stream.wait_event(e)
        with torch.cuda.stream(stream):
            graphs[b].replay()
            done[b].record(stream)
        for stm, dst, src, e in ((down[0], hy[b], dy[b], y_out[b]),
                                 (down[1], hgy[b], dgy[b], g_out[b])):
            stm.wait_event(done[b])
            with torch.cuda.stream(stm):
                dst.copy_(src, non_blocking=True)
                e.record(stm)

    steps = max(3, min(args.steps, 50))
    for s in range(3):
        one(s)
    torch.cuda.synchronize()
    barrier(world)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for s in range(steps):
        one(s)
    for e in y_out + g_out:
        stream.wait_event(e)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    secs = e0.elapsed_time(e1) / 1e3
    units, secs = aggregate(st.input_bytes * steps, secs, world, device)
    return {"value": round(units / secs / 1e9, 2), "unit": UNIT,
            "h2d_bytes_per_step": 2 * 4 * R * L, "d2h_bytes_per_step": 2 * 4 * R * L,
            "steps": steps, "api": "python binding calls of one step captured into a CUDA "
            "graph per input slot; per step two H2D copies from pinned memory and two D2H "
            "copies of results on copy streams, pipelined over two slots"}


def time_op(fn, stream, flush, reps=8):
    """Device time (ms) of one launch of fn on cold inputs, inside a CUDA graph: a graph of
    reps x (L2 flush, launch) against a graph of the reps flushes alone, the difference
    divided by reps (median of three), so that no event sits next to the launch."""
    sink = torch.empty((), dtype=torch.int64, device=flush.device)

    def fl():
        flush.fill_(1)
        torch.sum(flush.view(torch.int64), dim=0, out=sink)

    with torch.cuda.stream(stream):
        fn()
        fl()
        stream.synchronize()
        g1 = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g1, stream=stream):
            for _ in range(reps):
                fl()
                fn()
        g0 = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g0, stream=stream):
            for _ in range(reps):
                fl()

        def run(g):
            g.replay()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            g.replay()
            b.record(stream)
            stream.synchronize()
            return a.elapsed_time(b)

        d = [run(g1) - run(g0) for _ in range(3)]
    return max(statistics.median(d) / reps, 1e-4)


def measure_operators(mpc, synth, device, stream, peak):
    """Every operator of the path on its own workload: GB/s of algorithmic bytes and the
    fraction of HBM bandwidth."""
    out = {}
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=device)

    def rec(name, ms, nbytes):
        gbs = nbytes / (ms / 1e3) / 1e9
        out[name] = {"us": round(ms * 1e3, 2), "GBps": round(gbs, 1), "frac": round(gbs / peak, 4),
                     "MB": round(nbytes / 1e6, 2)}

    # small CNN boundary: Top10% and 8-bit
    x = synth.relu_normal((32, 16384), 0, device)
    k = synth.k_of(16384, 10)
    v, i = mpc.mpc_topk_compress(x, k)
    y = torch.empty_like(x)
    rec("topk_compress 32x16384 K=10%", time_op(lambda: mpc.mpc_topk_compress(x, k, v, i), stream, flush),
        algorithmic_bytes(32, 16384, k=k, op="topk"))
    rec("topk_decompress 32x16384 K=10%", time_op(lambda: mpc.mpc_topk_decompress(v, i, 16384, y=y), stream, flush),
        algorithmic_bytes(32, 16384, k=k, op="topk_decompress"))
    g1 = synth.normal((32, 16384), 1, device, std=1e-3)
    c1, s1, m1 = mpc.mpc_quant_compress(g1, 8)
    rec("quant_compress 32x16384 8-bit", time_op(lambda: mpc.mpc_quant_compress(g1, 8, codes=c1, scale=s1, minv=m1), stream, flush),
        algorithmic_bytes(32, 16384, bits=8, op="quant"))
    rec("quant_decompress 32x16384 8-bit", time_op(lambda: mpc.mpc_quant_decompress(c1, s1, m1, 16384, 8, y=y), stream, flush),
        algorithmic_bytes(32, 16384, bits=8, op="dequant"))
    del g1
    # index reuse at the CNN stage boundary: gradient values at the activation's Top10%
    xg = synth.relu_normal((R, L), 3, device)
    gg = synth.normal((R, L), 4, device, std=1e-3)
    kg = synth.k_of(L, 10)
    _, ig = mpc.mpc_topk_compress(xg, kg)
    vg = mpc.mpc_topk_gather(gg, ig)
    rec("topk_gather %dx%d K=10%%" % (R, L), time_op(lambda: mpc.mpc_topk_gather(gg, ig, vals=vg), stream, flush),
        algorithmic_bytes(R, L, k=kg, op="topk_gather"))
    del xg, gg
    # EF-mixed at the CNN stage boundary, Top10% (two selections and four small steps)
    xm = synth.relu_normal((R, L), 5, device)
    em = torch.zeros_like(xm)
    km = synth.k_of(L, 10)
    vm, im = mpc.mpc_efmix_topk_compress(xm, em, km)
    wsm = torch.empty(mpc.mpc_efmix_workspace_bytes(R, L, km), dtype=torch.uint8, device=device)
    rec("efmix_topk_compress %dx%d K=10%%" % (R, L), time_op(lambda: mpc.mpc_efmix_topk_compress(xm, em, km, vm, im, ws=wsm), stream, flush),
        algorithmic_bytes(R, L, k=km, op="efmix_topk"))
    del xm, em, wsm
    # LM boundary: EF21 Top10% per token, 4-bit
    xl = synth.lm_hidden(0, device)
    gl = torch.zeros_like(xl)
    kl = synth.k_of(768, 10)
    vl, il = mpc.mpc_ef21_topk_compress(xl, gl, kl)
    rec("ef21_topk_compress 8192x768 K=10%", time_op(lambda: mpc.mpc_ef21_topk_compress(xl, gl, kl, vl, il), stream, flush),
        algorithmic_bytes(8192, 768, k=kl, op="delta_topk"))
    cq, sq, mq = mpc.mpc_quant_compress(xl, 4)
    yl = torch.empty_like(xl)
    rec("quant_compress 8192x768 4-bit", time_op(lambda: mpc.mpc_quant_compress(xl, 4, codes=cq, scale=sq, minv=mq), stream, flush),
        algorithmic_bytes(8192, 768, bits=4, op="quant"))
    rec("quant_decompress 8192x768 4-bit", time_op(lambda: mpc.mpc_quant_decompress(cq, sq, mq, 768, 4, y=yl), stream, flush),
        algorithmic_bytes(8192, 768, bits=4, op="dequant"))
    # fw4-bw6: 6-bit codes of the transformer boundary's gradient (straddling words)
    g6 = synth.normal((8192, 768), 5, device, std=1e-4)
    c6, s6, m6 = mpc.mpc_quant_compress(g6, 6)
    rec("quant_compress 8192x768 6-bit", time_op(lambda: mpc.mpc_quant_compress(g6, 6, codes=c6, scale=s6, minv=m6), stream, flush),
        algorithmic_bytes(8192, 768, bits=6, op="quant"))
    rec("quant_decompress 8192x768 6-bit", time_op(lambda: mpc.mpc_quant_decompress(c6, s6, m6, 768, 6, y=yl), stream, flush),
        algorithmic_bytes(8192, 768, bits=6, op="dequant"))
    del g6
    del xl, gl, yl
    # AQ-SGD boundary: 8 GiB buffer, 16 ids, Top30%
    S, rps, La = 4096, 512, 1024
    buf = synth.normal((S, rps, La), 0, device)
    ids = synth.sample_ids(S, 16, 1, device)
    xa = buf[ids] + 0.05 * torch.randn((16, rps, La), device=device)
    ka = synth.k_of(La, 30)
    va, ia = mpc.mpc_aqsgd_compress(xa, buf, ids, ka)
    rec("aqsgd_compress 16x512x1024 K=30%", time_op(lambda: mpc.mpc_aqsgd_compress(xa, buf, ids, ka, va, ia), stream, flush),
        algorithmic_bytes(16 * rps, La, k=ka, op="delta_topk"))
    rec("aqsgd_decompress 16x512x1024 K=30%", time_op(lambda: mpc.mpc_aqsgd_decompress(va, ia, buf, ids), stream, flush),
        algorithmic_bytes(16 * rps, La, k=ka, op="aqsgd_decompress"))
    # the same boundary with 4-bit quantisation of the change (§2.5 with §2.2's quantiser)
    wsq = torch.empty(mpc.mpc_aqsgd_quant_workspace_bytes(16, rps, La, 4), dtype=torch.uint8,
                      device=device)
    cqa, sqa, mqa = mpc.mpc_aqsgd_quant_compress(xa, buf, ids, 4, ws=wsq)
    rec("aqsgd_quant_compress 16x512x1024 4-bit", time_op(lambda: mpc.mpc_aqsgd_quant_compress(xa, buf, ids, 4, codes=cqa, scale=sqa, minv=mqa, ws=wsq), stream, flush),
        algorithmic_bytes(16 * rps, La, bits=4, op="aqsgd_quant"))
    rec("aqsgd_quant_decompress 16x512x1024 4-bit", time_op(lambda: mpc.mpc_aqsgd_quant_decompress(cqa, sqa, mqa, buf, ids, 4), stream, flush),
        algorithmic_bytes(16 * rps, La, bits=4, op="aqsgd_dequant_add"))
    del buf, xa, wsq
    torch.cuda.empty_cache()
    # bandwidth sweep point: one 1 GiB tensor
    N = 1 << 28
    xs = synth.normal((N,), 28, device)
    for Ls in (768, 4096, 65536):
        Rs = N // Ls
        xv = xs[: Rs * Ls].view(Rs, Ls)
        for pct in (1, 10, 50):
            ks = synth.k_of(Ls, pct)
            vs, is_ = mpc.mpc_topk_compress(xv, ks)
            rec("topk_compress 2^28 L=%d K=%d%%" % (Ls, pct), time_op(lambda: mpc.mpc_topk_compress(xv, ks, vs, is_), stream, flush),
                algorithmic_bytes(Rs, Ls, k=ks, op="topk"))
            if pct == 10:
                gvs = mpc.mpc_topk_gather(xv, is_)
                rec("topk_gather 2^28 L=%d K=10%%" % Ls, time_op(lambda: mpc.mpc_topk_gather(xv, is_, vals=gvs), stream, flush),
                    algorithmic_bytes(Rs, Ls, k=ks, op="topk_gather"))
                del gvs
                ys = torch.empty_like(xv)
                rec("topk_decompress 2^28 L=%d K=10%%" % Ls, time_op(lambda: mpc.mpc_topk_decompress(vs, is_, Ls, y=ys), stream, flush),
                    algorithmic_bytes(Rs, Ls, k=ks, op="topk_decompress"))
                es = torch.zeros_like(xv)
                rec("ef_topk_compress 2^28 L=%d K=10%%" % Ls, time_op(lambda: mpc.mpc_ef_topk_compress(xv, es, ks, vs, is_), stream, flush),
                    algorithmic_bytes(Rs, Ls, k=ks, op="ef_topk"))
                del ys, es
            del vs, is_
        for b in BITS + (6,):
            cq, sq, mq = mpc.mpc_quant_compress(xv, b)
            rec("quant_compress 2^28 L=%d %d-bit" % (Ls, b), time_op(lambda: mpc.mpc_quant_compress(xv, b, codes=cq, scale=sq, minv=mq), stream, flush),
                algorithmic_bytes(Rs, Ls, bits=b, op="quant"))
            if b == 6:
                ys = torch.empty_like(xv)
                rec("quant_decompress 2^28 L=%d 6-bit" % Ls, time_op(lambda: mpc.mpc_quant_decompress(cq, sq, mq, Ls, 6, y=ys), stream, flush),
                    algorithmic_bytes(Rs, Ls, bits=6, op="dequant"))
                del ys
            if b == 4:
                rec("quant_compress 2^28 L=%d 4-bit stochastic" % Ls, time_op(lambda: mpc.mpc_quant_compress(xv, 4, True, 7, codes=cq, scale=sq, minv=mq), stream, flush),
                    algorithmic_bytes(Rs, Ls, bits=4, op="quant"))
                ys = torch.empty_like(xv)
                rec("quant_decompress 2^28 L=%d 4-bit" % Ls, time_op(lambda: mpc.mpc_quant_decompress(cq, sq, mq, Ls, 4, y=ys), stream, flush),
                    algorithmic_bytes(Rs, Ls, bits=4, op="dequant"))
                del ys
    del xs
    torch.cuda.empty_cache()
    st = mpc.mpc_get_status(stream)
    if st != 0:
        raise RuntimeError("device status %d: %s" % (st, mpc.mpc_last_error()))
    return out


# ---------------------------------------------------------------------------------------
# CPU oracle (the reference arm and the cpu_baseline key)
# ---------------------------------------------------------------------------------------

class OracleStep:
    """The same boundary step on SAMPLE_ROWS of the 128 rows, computed by the oracle."""

    def __init__(self, seed: int = 0):
        import oracle
        from paper_2401_07788_gb300 import synth

        self.oracle = oracle
        self.lib = oracle.load()
        x = synth.relu_normal((R, L), seed, "cpu")[:SAMPLE_ROWS].numpy().copy()
        g = synth.normal((R, L), 1000 + 100 * seed, "cpu", std=1e-3)[:SAMPLE_ROWS].numpy().copy()
        self.x, self.g = x, g
        self.ks = {p: synth.k_of(L, p) for p in TOPK_PCTS}
        self.errs = {p: np.zeros_like(x) for p in TOPK_PCTS}
        self.seed = seed
        self.input_bytes = 9 * 4 * SAMPLE_ROWS * L

    def run(self, step: int):
        o = self.oracle
        for p in TOPK_PCTS:
            v, i = o.ef_topk_compress(self.x, self.errs[p], self.ks[p], self.lib)
            o.topk_decompress(v, i, L, self.lib)
        for b in BITS:
            for sr in (False, True):
                c, s, m = o.quant_compress(self.g, b, sr, (self.seed << 32) | step, self.lib)
                o.quant_decompress(c, s, m, L, b, self.lib)


def cpu_baseline(budget_s: float = 10.0):
    st = OracleStep(0)
    st.run(0)
    n, t0 = 0, time.perf_counter()
    while time.perf_counter() - t0 < budget_s or n < 2:
        st.run(n)
        n += 1
    secs = time.perf_counter() - t0
    return {"value": round(st.input_bytes * n / secs / 1e9, 4), "unit": UNIT, "cores": 1,
            "kind": "oracle", "sample": "%d of %d rows of the step, %d steps in %.1f s"
            % (SAMPLE_ROWS, R, n, secs), "cpu": cpu_name()}


def cpu_name():
    try:
        for ln in open("/proc/cpuinfo"):
            if ln.lower().startswith(("model name", "cpu part")):
                return ln.split(":", 1)[1].strip()
    except OSError:
        pass
    return os.uname().machine


def run_reference(args, rank, world):
    if rank != 0:
        return
    st = OracleStep(0)
    for w in range(args.warmup):
        st.run(w)
    t0 = time.perf_counter()
    for s in range(args.steps):
        st.run(s)
    secs = time.perf_counter() - t0
    value = st.input_bytes * args.steps / secs / 1e9
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": UNIT,
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(secs * 1e3 / args.steps, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": WORKLOAD, "rows": R, "row_len": L,
                   "topk_percents": list(TOPK_PCTS), "bits": list(BITS),
                   "sample_rows": SAMPLE_ROWS},
        "cpu_baseline": {"value": round(value, 4), "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": "%d of %d rows of each step" % (SAMPLE_ROWS, R),
                         "cpu": cpu_name()},
        "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_sweep():
    """The size sweep of the bandwidth study: N = 2^20..2^30 N(0,1) entries as rows of
    L in {768, 4096, 65536, N} (N itself only up to 2^26, the on-chip row path's reach
    being 65536 and the grid path's workspace growing with the row); TopK and EF-TopK at
    K = 1, 10, 50 %, 2/4/8-bit quantisation and 4-bit dequantisation, each launch timed
    inside a CUDA graph on cold inputs as in `operators`."""
    import paper_2401_07788_gb300 as mpc
    from paper_2401_07788_gb300 import synth

    device = torch.device("cuda", 0)
    torch.cuda.set_device(device)
    stream = torch.cuda.Stream(device)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=device)
    peak, _ = hbm_peak()
    table = []
    for log2n in range(20, 31):
        N = 1 << log2n
        xs = synth.normal((N,), log2n, device)
        for Ls in (768, 4096, 65536) + ((N,) if log2n <= 26 else ()):
            Rs = N // Ls
            if Rs < 1:
                continue
            xv = xs[: Rs * Ls].view(Rs, Ls)
            entries = []
            for pct in (1, 10, 50):
                ks = synth.k_of(Ls, pct)
                vs, is_ = mpc.mpc_topk_compress(xv, ks)
                ws = None
                need = mpc.mpc_topk_workspace_bytes(Rs, Ls, ks)
                if need:
                    ws = torch.empty(need, dtype=torch.uint8, device=device)
                entries.append(("topk K=%d%%" % pct, time_op(lambda: mpc.mpc_topk_compress(xv, ks, vs, is_, ws=ws), stream, flush),
                                algorithmic_bytes(Rs, Ls, k=ks, op="topk")))
                es = torch.zeros_like(xv)
                entries.append(("ef_topk K=%d%%" % pct, time_op(lambda: mpc.mpc_ef_topk_compress(xv, es, ks, vs, is_, ws=ws), stream, flush),
                                algorithmic_bytes(Rs, Ls, k=ks, op="ef_topk")))
                del es, vs, is_, ws
            for b in ((2, 4, 8) if Ls <= 0x7fffffff // 32 else ()):  # the quantiser's row limit
                cq, sq, mq = mpc.mpc_quant_compress(xv, b)
                entries.append(("quant %d-bit" % b, time_op(lambda: mpc.mpc_quant_compress(xv, b, codes=cq, scale=sq, minv=mq), stream, flush),
                                algorithmic_bytes(Rs, Ls, bits=b, op="quant")))
                if b == 4:
                    ys = torch.empty_like(xv)
                    entries.append(("dequant 4-bit", time_op(lambda: mpc.mpc_quant_decompress(cq, sq, mq, Ls, 4, y=ys), stream, flush),
                                    algorithmic_bytes(Rs, Ls, bits=4, op="dequant")))
                    del ys
                del cq, sq, mq
            for name, ms, nbytes in entries:
                gbs = nbytes / (ms / 1e3) / 1e9
                table.append({"log2n": log2n, "row_len": Ls, "op": name, "us": round(ms * 1e3, 2),
                              "GBps": round(gbs, 1), "frac": round(gbs / peak, 4)})
        del xs
        torch.cuda.empty_cache()
    st = mpc.mpc_get_status(stream)
    if st != 0:
        raise RuntimeError("device status %d: %s" % (st, mpc.mpc_last_error()))
    print(json.dumps({"sweep": table, "peak": peak, "unit": "GB/s", "timing": "each launch "
                      "inside a CUDA graph on cold inputs (flush-and-launch graph against a "
                      "flush-only graph)"}), flush=True)


def main():
    args = parse_args()
    rank, local, world = dist_env()
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if args.sweep:
        if rank == 0:
            run_sweep()
        return
    run_ours(args, rank, local, world)
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


if __name__ == "__main__":
    main()
