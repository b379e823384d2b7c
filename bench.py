#!/usr/bin/env python3
"""Benchmark of libmpcomp: compress+decompress GB/s (input bytes) and the fraction of HBM
bandwidth per operator, on one GB300.

Headline workload: the bandwidth sweep at its largest size, one N(0,1) fp32 tensor of
2^30 entries (4 GiB), reshaped to rows of 768, 4096 and 65536 entries and to one
whole-tensor row.  One step runs, for each of the four row lengths, every
compress+decompress pair of the sweep on that step's tensor:
  TopK at K = 1, 10, 50 %, each followed by TopK decompression;
  error-feedback TopK at K = 1, 10, 50 % (one error buffer per row length and K, carried
  across steps), each followed by decompression of its payload;
  2/4/8-bit min-max quantisation (round to nearest), each followed by dequantisation.
That is 36 pairs (72 library calls) per step, in order on one stream; two input tensors
alternate from step to step.  value = 36 x 4 x 2^30 input bytes per step / device time of
the step (CUDA events on the stream, max over ranks).  Every input is 4 GiB, far larger
than the 126 MB L2, so no L2 flush is needed between steps.  An event after every call
gives each call's duration inside the timed region; `roofline` reports the call with the
largest share of the step: its algorithmic bytes (inputs and buffers read once, payload
and buffers written once) / its average duration, against the measured copy bandwidth.
`e2e` runs the same steps through the same calls with the input tensor copied from
pinned host memory and the last dequantised tensor copied back every step (pipelined over
two slots).  `per_op` lists every call of the step.

Secondary keys: `cnn_boundary_step`, the CNN stage boundary [128,128,16,16] (EF-TopK at
5/10/30 % and 2/4/8-bit quantisation, nearest and stochastic, with their
decompressions; one CUDA graph per step); `whole_tensor`, whole-tensor rows of 2^27,
2^28 and 2^29 entries; `operators`, every operator on its own workload (the small CNN,
transformer and AQ-SGD boundaries, index reuse, EF-mixed, stochastic and 6-bit codes, and
256 rows of 2^20 entries through the grid path's batches of rows).

`--impl reference` and `cpu_baseline` time the CPU oracle (single-threaded C) on a
bounded sample of the same step: a few rows of each row length and a whole-tensor row of
2^20 entries.
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
LOG2N = 30
SWEEP_LENS = (768, 4096, 65536, None)  # None: the whole tensor as one row
SWEEP_PCTS = (1, 10, 50)
SWEEP_BITS = (2, 4, 8)
# the CNN stage boundary (secondary key)
R, L = 128, 32768
TOPK_PCTS = (5, 10, 30)
BITS = (2, 4, 8)
POOL = 4


def parse_args():
    p = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=("ours", "reference"), default="ours")
    p.add_argument("--log2n", type=int, default=LOG2N,
                   help="entries of the headline tensor, log2 (the workload is 2^30)")
    p.add_argument("--no-operators", action="store_true", help="skip the per-operator table")
    p.add_argument("--no-secondary", action="store_true",
                   help="skip the CNN-boundary step and the whole-tensor table")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--profile-call", default="",
                   help="for ncu captures: run only these calls of the sweep step (comma-separated "
                        "names as in the per_op table, in order), warm-up and timed steps alike, "
                        "and print one line saying what ran instead of the benchmark line")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cnn-steps", type=int, default=200)
    p.add_argument("--branches", type=int, default=6, choices=(1, 2, 3, 5, 6, 9),
                   help="concurrent streams inside the CNN-boundary step graph")
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
# algorithmic bytes and the kernels behind each call
# ---------------------------------------------------------------------------------------

def algorithmic_bytes(R_, L_, k=None, bits=None, op=""):
    """Minimum HBM bytes of one call: inputs and buffers read once, payload and buffers
    written once (the buffer of EF21 / AQ-SGD counted as read and written in full)."""
    N = R_ * L_
    if op in ("ef_topk", "delta_topk", "efmix_topk"):  # x, buffer read; buffer, payload written
        return 12 * N + 8 * k * R_
    if op == "topk":
        return 4 * N + 8 * k * R_
    if op == "topk_decompress":
        return 8 * k * R_ + 4 * N
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


ROW_PATH_MAX = 65536  # longest row of the on-chip TopK and single-pass quantisation kernels


def kernels_of(op: str, L_: int) -> list:
    """The library kernels one call launches, in order (the launch count is their number)."""
    if op in ("topk", "ef_topk"):
        if L_ <= 1024:
            return ["topk_warp_kernel"]
        if L_ <= 8192:
            return ["topk_band_kernel"]
        if L_ <= ROW_PATH_MAX:
            return ["topk_lrow_kernel"]  # 16-byte aligned rows (the sweep's are)
        return (["g_init", "w_sample", "w_spick", "w_pass1", "w_pick1", "w_bin2", "w_select2",
                 "w_mark", "g_sample"] + ["g_hist", "g_pick"] * 4
                + ["g_count", "g_select", "w_scan1", "w_scan2", "g_write3", "g_wlist"])
    if op == "topk_decompress":
        return ["topk_decompress_tiles_kernel"]
    if op == "quant":
        if L_ <= 2048:
            return ["quant_warp_kernel"]
        if L_ <= 4096:
            return ["quant_rows4_kernel"]
        if L_ <= ROW_PATH_MAX:
            return ["quant_cta_kernel"]
        return ["minmax_init_kernel", "quant_minmax_kernel", "quant_cta_kernel"]
    if op == "dequant":
        return ["dequant_rows_kernel"]
    raise ValueError(op)


# ---------------------------------------------------------------------------------------
# the headline step: the bandwidth sweep at 2^30 entries
# ---------------------------------------------------------------------------------------

def headline_call_names(log2n: int = LOG2N) -> list:
    """Names of the calls of one headline step, in launch order (no device needed)."""
    N = 1 << log2n
    names = []
    for Ls in SWEEP_LENS:
        tag = "L=%s" % ("N" if Ls is None else Ls)
        for feedback in (False, True):
            for p in SWEEP_PCTS:
                names.append(("ef_topk_compress %s K=%d%%" if feedback else "topk_compress %s K=%d%%")
                             % (tag, p))
                names.append("topk_decompress %s K=%d%%%s" % (tag, p, " (EF)" if feedback else ""))
        for b in SWEEP_BITS:
            names += ["quant_compress %s %d-bit" % (tag, b), "quant_decompress %s %d-bit" % (tag, b)]
    assert N > 0
    return names


class Call:
    __slots__ = ("name", "op", "L", "fn", "nbytes", "in_bytes", "kernels")

    def __init__(self, name, op, L_, fn, nbytes, in_bytes):
        self.name, self.op, self.L, self.fn = name, op, L_, fn
        self.nbytes, self.in_bytes = nbytes, in_bytes
        self.kernels = kernels_of(op, L_)


class SweepStep:
    """Buffers and the 72 calls of one step of the sweep at N entries.  Every call takes
    the step's input tensor x (N entries) and the dense output y (N entries), so the same
    calls serve the device-resident and the end-to-end runs."""

    def __init__(self, mpc, synth, device, log2n: int, seed: int):
        self.mpc = mpc
        N = 1 << log2n
        self.N = N
        self.xs = [synth.normal((N,), 1000 * seed + log2n + 17 * t, device) for t in range(2)]
        self.y = torch.empty(N, device=device)
        self.seed = seed
        shapes = []
        for Ls in SWEEP_LENS:
            Lr = N if Ls is None else Ls
            shapes.append((N // Lr, Lr))
        self.shapes = shapes
        max_pay = max(Rr * synth.k_of(Lr, p) for Rr, Lr in shapes for p in SWEEP_PCTS)
        self.vals = torch.empty(max_pay, device=device)
        self.idx = torch.empty(max_pay, dtype=torch.int32, device=device)
        max_words = max(mpc.mpc_quant_codes_words(Rr, Lr, b) for Rr, Lr in shapes for b in SWEEP_BITS)
        self.codes = torch.empty(max_words, dtype=torch.int32, device=device)
        max_rows = max(Rr for Rr, _ in shapes)
        self.scale = torch.empty(max_rows, device=device)
        self.minv = torch.empty(max_rows, device=device)
        tws = max(mpc.mpc_topk_workspace_bytes(Rr, Lr, synth.k_of(Lr, p))
                  for Rr, Lr in shapes for p in SWEEP_PCTS)
        qws = max(mpc.mpc_quant_workspace_bytes(Rr, Lr, b) for Rr, Lr in shapes for b in SWEEP_BITS)
        self.tws = torch.empty(max(tws, 256), dtype=torch.uint8, device=device)
        self.qws = torch.empty(max(qws, 256), dtype=torch.uint8, device=device)
        self.errs = {}
        self.calls = []
        m = mpc
        for Rr, Lr in shapes:
            tag = "L=%s" % ("N" if Lr == N else Lr)
            n = Rr * Lr
            for feedback in (False, True):
                for p in SWEEP_PCTS:
                    k = synth.k_of(Lr, p)
                    v = self.vals[: Rr * k].view(Rr, k)
                    i = self.idx[: Rr * k].view(Rr, k)
                    if feedback:
                        e = torch.zeros((Rr, Lr), device=device)
                        self.errs[(Lr, p)] = e
                        fn = (lambda x, y, Rr=Rr, Lr=Lr, k=k, v=v, i=i, e=e: m.mpc_ef_topk_compress(
                            x[: Rr * Lr].view(Rr, Lr), e, k, v, i, ws=self.tws))
                        self.calls.append(Call("ef_topk_compress %s K=%d%%" % (tag, p), "ef_topk", Lr,
                                               fn, algorithmic_bytes(Rr, Lr, k=k, op="ef_topk"), 4 * n))
                    else:
                        fn = (lambda x, y, Rr=Rr, Lr=Lr, k=k, v=v, i=i: m.mpc_topk_compress(
                            x[: Rr * Lr].view(Rr, Lr), k, v, i, ws=self.tws))
                        self.calls.append(Call("topk_compress %s K=%d%%" % (tag, p), "topk", Lr, fn,
                                               algorithmic_bytes(Rr, Lr, k=k, op="topk"), 4 * n))
                    fn = (lambda x, y, Rr=Rr, Lr=Lr, v=v, i=i: m.mpc_topk_decompress(
                        v, i, Lr, y=y[: Rr * Lr].view(Rr, Lr)))
                    self.calls.append(Call("topk_decompress %s K=%d%%%s" % (tag, p, " (EF)" if feedback else ""),
                                           "topk_decompress", Lr, fn,
                                           algorithmic_bytes(Rr, Lr, k=k, op="topk_decompress"), 0))
            for b in SWEEP_BITS:
                W = m.mpc_quant_codes_words(Rr, Lr, b) // Rr
                c = self.codes[: Rr * W].view(Rr, W)
                sc, mn = self.scale[:Rr], self.minv[:Rr]
                fn = (lambda x, y, Rr=Rr, Lr=Lr, b=b, c=c, sc=sc, mn=mn: m.mpc_quant_compress(
                    x[: Rr * Lr].view(Rr, Lr), b, codes=c, scale=sc, minv=mn, ws=self.qws))
                self.calls.append(Call("quant_compress %s %d-bit" % (tag, b), "quant", Lr, fn,
                                       algorithmic_bytes(Rr, Lr, bits=b, op="quant"), 4 * n))
                fn = (lambda x, y, Rr=Rr, Lr=Lr, b=b, c=c, sc=sc, mn=mn: m.mpc_quant_decompress(
                    c, sc, mn, Lr, b, y=y[: Rr * Lr].view(Rr, Lr)))
                self.calls.append(Call("quant_decompress %s %d-bit" % (tag, b), "dequant", Lr, fn,
                                       algorithmic_bytes(Rr, Lr, bits=b, op="dequant"), 0))
        assert [c.name for c in self.calls] == headline_call_names(log2n)
        self.input_bytes = sum(c.in_bytes for c in self.calls)
        self.launches = sum(len(c.kernels) for c in self.calls)

    def run(self, x, y, events=None):
        for j, c in enumerate(self.calls):
            c.fn(x, y)
            if events is not None:
                events[j].record()


def run_profile_calls(args, st, mpc, device):
    """Only the named calls of the sweep step, in the given order, for warm-up + timed steps
    (a profiler then picks the launches it wants); no timing is reported."""
    by_name = {c.name: c for c in st.calls}
    names = [s.strip() for s in args.profile_call.split(",") if s.strip()]
    missing = [s for s in names if s not in by_name]
    if missing:
        raise SystemExit("unknown call(s): %s" % ", ".join(missing))
    stream = torch.cuda.Stream(device)
    with torch.cuda.stream(stream):
        for s in range(max(1, args.warmup) + args.steps):
            for n in names:
                by_name[n].fn(st.xs[s % 2], st.y)
    stream.synchronize()
    status = mpc.mpc_get_status(stream)
    if status != 0:
        raise RuntimeError("device status %d: %s" % (status, mpc.mpc_last_error()))
    print(json.dumps({"profile_call": names, "log2n": args.log2n,
                      "runs": max(1, args.warmup) + args.steps,
                      "launches_per_run": sum(len(by_name[n].kernels) for n in names)}), flush=True)


def run_headline(args, rank, local, world):
    import paper_2401_07788_gb300 as mpc
    from paper_2401_07788_gb300 import synth

    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    init_dist(world, "nccl")
    mpc.lib()
    st = SweepStep(mpc, synth, device, args.log2n, rank % 10)
    if args.profile_call:
        run_profile_calls(args, st, mpc, device)
        return
    n_calls = len(st.calls)
    stream = torch.cuda.Stream(device)
    with torch.cuda.stream(stream):
        for w in range(max(1, args.warmup)):
            st.run(st.xs[w % 2], st.y)
    stream.synchronize()
    status = mpc.mpc_get_status(stream)
    if status != 0:
        raise RuntimeError("device status %d: %s" % (status, mpc.mpc_last_error()))

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(n_calls)] for _ in range(args.steps)]
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    barrier(world)
    torch.cuda.synchronize()
    sampler = ClockSampler(local)
    sampler.__enter__()
    t0 = time.perf_counter()
    with torch.cuda.stream(stream):
        for s in range(args.steps):
            starts[s].record(stream)
            st.run(st.xs[s % 2], st.y, evs[s])
    stream.synchronize()
    wall = time.perf_counter() - t0
    sampler.__exit__(None, None, None)
    clocks = sampler.summary()
    barrier(world)
    status = mpc.mpc_get_status(stream)
    if status != 0:
        raise RuntimeError("device status %d: %s" % (status, mpc.mpc_last_error()))
    op_ms = [0.0] * n_calls
    dev_ms = 0.0
    for s in range(args.steps):
        prev = starts[s]
        for j in range(n_calls):
            op_ms[j] += prev.elapsed_time(evs[s][j])
            prev = evs[s][j]
        dev_ms += starts[s].elapsed_time(evs[s][-1])
    units, secs = aggregate(st.input_bytes * args.steps, dev_ms / 1e3, world, device)
    value = units / secs / 1e9

    peak, peak_kind = hbm_peak()
    per_op = {}
    for j, c in enumerate(st.calls):
        us = op_ms[j] / args.steps * 1e3
        gbs = c.nbytes / (us / 1e6) / 1e9
        per_op[c.name] = {"us": round(us, 1), "GBps": round(gbs, 1), "frac": round(gbs / peak, 4),
                          "launches": len(c.kernels)}
    dom = max(range(n_calls), key=lambda j: op_ms[j])
    c = st.calls[dom]
    avg_ms = op_ms[dom] / args.steps
    achieved = c.nbytes / (avg_ms / 1e3) / 1e9
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4),
                "traffic": recorded_traffic(c.name),
                "op": c.name, "kernels": sorted(set(c.kernels)), "launches_per_call": len(c.kernels),
                "algorithmic_bytes": c.nbytes, "avg_call_us": round(avg_ms * 1e3, 1),
                "share_of_step": round(op_ms[dom] / max(sum(op_ms), 1e-9), 4),
                "peak_source": peak_kind + " (MEASURED_PEAKS.json hbm_gbs, copy bandwidth)"
                if peak_kind == "measured" else peak_kind,
                "timing": "CUDA events on the launching stream before and after the call, "
                          "inside the timed steps, averaged over the steps"}

    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, st, stream, world, device)

    cnn = whole = operators = None
    if not args.no_secondary:
        cnn = run_cnn_step(args, mpc, synth, device, world)
        if rank == 0:
            whole = measure_whole_tensor(mpc, synth, device, stream, peak)
    if not args.no_operators and rank == 0:
        operators = measure_operators(mpc, synth, device, stream, peak)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(budget_s=10.0)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(secs * 1e3 / args.steps, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": "bandwidth sweep at 2^%d entries: one N(0,1) fp32 tensor of "
                                   "%d entries as rows of 768, 4096, 65536 and one whole-tensor row"
                                   % (args.log2n, st.N),
                       "entries": st.N, "row_lens": [Lr for _, Lr in st.shapes],
                       "rows": [Rr for Rr, _ in st.shapes],
                       "topk_percents": list(SWEEP_PCTS), "ef_topk_percents": list(SWEEP_PCTS),
                       "bits": list(SWEEP_BITS), "rounding": "nearest",
                       "pairs_per_step": n_calls // 2, "calls_per_step": n_calls,
                       "input_bytes_per_step": st.input_bytes,
                       "l2": "no flush: every input is %d bytes, larger than the 126 MB L2" % (4 * st.N),
                       "parallelism": "replicas" if world > 1 else "single GPU"},
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": st.launches * args.steps, "clocks": clocks,
            "wall_s": round(wall, 3), "per_op": per_op,
            "cnn_boundary_step": cnn, "whole_tensor": whole, "operators": operators,
        }
        print(json.dumps(line), flush=True)


def run_e2e(args, st, stream, world, device):
    """The headline steps end to end: every step copies its input tensor from pinned host
    memory to the device and the last dequantised tensor back, inside the timed region,
    through the same calls.  Copies and compute are pipelined over two slots (step s+1's
    input goes up while step s computes and step s-1's result comes down), each copy on its
    own stream."""
    N = st.N
    hx = st.xs[0].cpu().pin_memory()
    hy = [torch.empty(N, pin_memory=True) for _ in range(2)]
    dx = [torch.empty(N, device=device) for _ in range(2)]
    dy = [torch.empty(N, device=device) for _ in range(2)]
    up, down = torch.cuda.Stream(device), torch.cuda.Stream(device)
    ev = lambda: [torch.cuda.Event() for _ in range(2)]  # noqa: E731
    x_in, done, y_out = ev(), ev(), ev()
    for e in done + y_out:
        e.record(stream)

    def one(s):
        b = s % 2
        up.wait_event(done[b])  # the slot's previous compute has read its input
        with torch.cuda.stream(up):
            dx[b].copy_(hx, non_blocking=True)
            x_in[b].record(up)
        stream.wait_event(x_in[b])
        stream.wait_event(y_out[b])  # the slot's previous result has been copied out
        with torch.cuda.stream(stream):
            st.run(dx[b], dy[b])
            done[b].record(stream)
        down.wait_event(done[b])
        with torch.cuda.stream(down):
            hy[b].copy_(dy[b], non_blocking=True)
            y_out[b].record(down)

    steps = max(2, min(args.steps, 4))
    one(0)
    torch.cuda.synchronize()
    barrier(world)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for s in range(steps):
        one(s)
    for e in y_out:
        stream.wait_event(e)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    secs = e0.elapsed_time(e1) / 1e3
    units, secs = aggregate(st.input_bytes * steps, secs, world, device)
    del dx, dy
    return {"value": round(units / secs / 1e9, 2), "unit": UNIT,
            "h2d_bytes_per_step": 4 * N, "d2h_bytes_per_step": 4 * N, "steps": steps,
            "api": "the step's 72 library calls through the Python binding; per step one H2D "
                   "copy of the input from pinned memory and one D2H copy of a result, on copy "
                   "streams, pipelined over two slots"}


def measure_whole_tensor(mpc, synth, device, stream, peak, log2ns=(27, 28, 29)):
    """Whole-tensor rows below the headline size: TopK and EF-TopK at K = 10 %, 4-bit
    quantisation and the decompressions, each call timed between events over 3 calls in a
    row (inputs of 512 MiB and more, larger than L2)."""
    out = {}

    def timed(fn, reps=3):
        with torch.cuda.stream(stream):
            fn()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for _ in range(reps):
                fn()
            b.record(stream)
            stream.synchronize()
        return a.elapsed_time(b) / reps

    def rec(name, ms, nbytes):
        gbs = nbytes / (ms / 1e3) / 1e9
        out[name] = {"us": round(ms * 1e3, 1), "GBps": round(gbs, 1), "frac": round(gbs / peak, 4)}

    for lg in log2ns:
        N = 1 << lg
        x = synth.normal((1, N), lg, device)
        k = synth.k_of(N, 10)
        ws = torch.empty(mpc.mpc_topk_workspace_bytes(1, N, k), dtype=torch.uint8, device=device)
        v, i = mpc.mpc_topk_compress(x, k, ws=ws)
        rec("topk_compress 2^%d K=10%%" % lg, timed(lambda: mpc.mpc_topk_compress(x, k, v, i, ws=ws)),
            algorithmic_bytes(1, N, k=k, op="topk"))
        y = torch.empty_like(x)
        rec("topk_decompress 2^%d K=10%%" % lg, timed(lambda: mpc.mpc_topk_decompress(v, i, N, y=y)),
            algorithmic_bytes(1, N, k=k, op="topk_decompress"))
        e = torch.zeros_like(x)
        rec("ef_topk_compress 2^%d K=10%%" % lg, timed(lambda: mpc.mpc_ef_topk_compress(x, e, k, v, i, ws=ws)),
            algorithmic_bytes(1, N, k=k, op="ef_topk"))
        del e, v, i, ws
        qws = torch.empty(mpc.mpc_quant_workspace_bytes(1, N, 4), dtype=torch.uint8, device=device)
        c, sc, mn = mpc.mpc_quant_compress(x, 4, ws=qws)
        rec("quant_compress 2^%d 4-bit" % lg, timed(lambda: mpc.mpc_quant_compress(x, 4, codes=c, scale=sc, minv=mn, ws=qws)),
            algorithmic_bytes(1, N, bits=4, op="quant"))
        rec("quant_decompress 2^%d 4-bit" % lg, timed(lambda: mpc.mpc_quant_decompress(c, sc, mn, N, 4, y=y)),
            algorithmic_bytes(1, N, bits=4, op="dequant"))
        del x, y, c, qws
        torch.cuda.empty_cache()
    st = mpc.mpc_get_status(stream)
    if st != 0:
        raise RuntimeError("device status %d: %s" % (st, mpc.mpc_last_error()))
    return out


# ---------------------------------------------------------------------------------------
# the CNN stage boundary (secondary key)
# ---------------------------------------------------------------------------------------

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


def run_cnn_step(args, mpc, synth, device, world):
    """The CNN stage boundary [128,128,16,16] (the round of every operator that workload
    sweeps, 18 library calls) as one CUDA graph per step, its nine independent
    compress+decompress pairs on concurrent branches (--branches); a 256 MiB buffer written
    then read before each step, outside the timed interval, takes the step's inputs out of
    L2.  The dominant call is timed over 200 calls in a row on cold input copies."""
    st = Step(mpc, synth, device, 0)
    n_ops = len(st.ops)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=device)
    sink = torch.empty((), dtype=torch.int64, device=device)
    stream = torch.cuda.Stream(device)
    side = [torch.cuda.Stream(device) for _ in range(args.branches - 1)]

    def flush_l2(i):
        flush.fill_(i & 0xff)
        torch.sum(flush.view(torch.int64), dim=0, out=sink)

    with torch.cuda.stream(stream):
        for w in range(2):
            st.launch(w % POOL, w)
            st.launch(w % POOL, w, side=side)
    stream.synchronize()
    assert mpc.mpc_get_status(stream) == 0, mpc.mpc_last_error()
    keep = []

    def capture(slot, **kw):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            st.launch(slot, slot, **kw)
        return g

    plain = [capture(slot, side=side) for slot in range(POOL)]
    evsets = [[torch.cuda.Event(enable_timing=True, external=True) for _ in range(n_ops)]
              for _ in range(POOL)]
    keep.append(evsets)
    evented = [capture(slot, events=evsets[slot]) for slot in range(POOL)]
    torch.cuda.synchronize()
    steps = args.cnn_steps

    def timed_pass(graphs, after_step=None):
        starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
        ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
        with torch.cuda.stream(stream):
            for w in range(max(3, args.warmup)):
                flush_l2(w)
                graphs[w % POOL].replay()
        stream.synchronize()
        barrier(world)
        with torch.cuda.stream(stream):
            for i in range(steps):
                flush_l2(i)
                starts[i].record(stream)
                graphs[i % POOL].replay()
                ends[i].record(stream)
                if after_step is not None and ((i + 1) % POOL == 0 or i == steps - 1):
                    stream.synchronize()
                    for j in range(i - (i % POOL), i + 1):
                        after_step(j, starts[j], ends[j])
        stream.synchronize()
        barrier(world)
        return sum(starts[i].elapsed_time(ends[i]) for i in range(steps)) / 1e3

    for p in TOPK_PCTS:
        st.errs[p].zero_()
    dev_s = timed_pass(plain)
    op_ms = [0.0] * n_ops

    def read_ops(j, start, end):
        prev = start
        for i, ev in enumerate(evsets[j % POOL]):
            op_ms[i] += prev.elapsed_time(ev)
            prev = ev

    timed_pass(evented, read_ops)
    dom = max(range(n_ops), key=lambda j: op_ms[j])
    dom_ms = time_back_to_back(st, dom, stream, flush_l2)
    status = mpc.mpc_get_status(stream)
    if status != 0:
        raise RuntimeError("device status %d: %s" % (status, mpc.mpc_last_error()))
    units, secs = aggregate(st.input_bytes * steps, dev_s, world, device)
    peak, _ = hbm_peak()
    name, nbytes = st.ops[dom]
    achieved = nbytes / (dom_ms / 1e3) / 1e9
    del plain, evented, keep, flush
    return {"workload": "CNN stage boundary [128,128,16,16] fp32, 128 rows x 32768",
            "value": round(units / secs / 1e9, 2), "unit": UNIT, "steps": steps,
            "ms_per_step": round(secs * 1e3 / steps, 4), "launches_per_step": n_ops,
            "step": "one CUDA graph per step (no event nodes inside); " + BRANCH_TEXT[args.branches],
            "l2": "256 MiB buffer written then read before each timed step, outside the timed "
                  "interval",
            "dominant": {"op": name, "avg_launch_us": round(dom_ms * 1e3, 2),
                         "achieved": round(achieved, 1), "frac": round(achieved / peak, 4),
                         "algorithmic_bytes": nbytes,
                         "timing": "200 launches in a row on its stream between two CUDA "
                                   "events, inputs cycling through 8 copies (twice the L2)"},
            "per_op_us": {st.ops[j][0]: round(op_ms[j] / steps * 1e3, 2) for j in range(n_ops)}}


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


# ---------------------------------------------------------------------------------------
# every operator on its own workload
# ---------------------------------------------------------------------------------------

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
    # sweep point of 2^28 entries: the calls the headline step does not make (index reuse,
    # stochastic rounding, 6-bit codes) at each row length
    N = 1 << 28
    xs = synth.normal((N,), 28, device)
    for Ls in (768, 4096, 65536):
        Rs = N // Ls
        xv = xs[: Rs * Ls].view(Rs, Ls)
        ks = synth.k_of(Ls, 10)
        vs, is_ = mpc.mpc_topk_compress(xv, ks)
        gvs = mpc.mpc_topk_gather(xv, is_)
        rec("topk_gather 2^28 L=%d K=10%%" % Ls, time_op(lambda: mpc.mpc_topk_gather(xv, is_, vals=gvs), stream, flush),
            algorithmic_bytes(Rs, Ls, k=ks, op="topk_gather"))
        gs = torch.zeros_like(xv)
        rec("ef21_topk_compress 2^28 L=%d K=10%%" % Ls, time_op(lambda: mpc.mpc_ef21_topk_compress(xv, gs, ks, vs, is_), stream, flush),
            algorithmic_bytes(Rs, Ls, k=ks, op="delta_topk"))
        del gvs, vs, is_, gs
        for b, sr in ((4, True), (8, True), (6, False)):
            cq, sq, mq = mpc.mpc_quant_compress(xv, b)
            rec("quant_compress 2^28 L=%d %d-bit %s" % (Ls, b, "stochastic" if sr else "nearest"),
                time_op(lambda: mpc.mpc_quant_compress(xv, b, sr, 7, codes=cq, scale=sq, minv=mq), stream, flush),
                algorithmic_bytes(Rs, Ls, bits=b, op="quant"))
            if b == 6:
                ys = torch.empty_like(xv)
                rec("quant_decompress 2^28 L=%d 6-bit" % Ls, time_op(lambda: mpc.mpc_quant_decompress(cq, sq, mq, Ls, 6, y=ys), stream, flush),
                    algorithmic_bytes(Rs, Ls, bits=6, op="dequant"))
                del ys
            del cq, sq, mq
    # many long rows (256 rows of 2^20 entries): the grid path's batches of rows
    Ll = 1 << 20
    Rl = N // Ll
    xl2 = xs.view(Rl, Ll)
    kl2 = synth.k_of(Ll, 10)
    wsl = torch.empty(mpc.mpc_topk_workspace_bytes(Rl, Ll, kl2), dtype=torch.uint8, device=device)
    vl2, il2 = mpc.mpc_topk_compress(xl2, kl2, ws=wsl)
    rec("topk_compress 2^28 L=2^20 K=10%", time_op(lambda: mpc.mpc_topk_compress(xl2, kl2, vl2, il2, wsl), stream, flush),
        algorithmic_bytes(Rl, Ll, k=kl2, op="topk"))
    el2 = torch.zeros_like(xl2)
    rec("ef_topk_compress 2^28 L=2^20 K=10%", time_op(lambda: mpc.mpc_ef_topk_compress(xl2, el2, kl2, vl2, il2, wsl), stream, flush),
        algorithmic_bytes(Rl, Ll, k=kl2, op="ef_topk"))
    del vl2, il2, el2, wsl, xl2
    del xs
    torch.cuda.empty_cache()
    st = mpc.mpc_get_status(stream)
    if st != 0:
        raise RuntimeError("device status %d: %s" % (st, mpc.mpc_last_error()))
    return out


# ---------------------------------------------------------------------------------------
# CPU oracle (the reference arm and the cpu_baseline key)
# ---------------------------------------------------------------------------------------

# Bounded sample of the headline step for the single-threaded oracle: entries per row
# length (whole rows of 768, 4096 and 65536 entries), and one whole-tensor row of 2^20.
ORACLE_SAMPLE = ((768, 1 << 17), (4096, 1 << 17), (65536, 1 << 17), (None, 1 << 20))


class OracleStep:
    """The headline step on the bounded sample, computed by the oracle: for each row length
    the same 18 calls (TopK and EF-TopK at 1/10/50 % with decompression, 2/4/8-bit
    quantisation with dequantisation)."""

    def __init__(self, seed: int = 0):
        import oracle
        from paper_2401_07788_gb300 import synth

        self.oracle = oracle
        self.lib = oracle.load()
        self.parts = []
        for Ls, n in ORACLE_SAMPLE:
            Lr = n if Ls is None else Ls
            Rr = n // Lr
            x = synth.normal((Rr, Lr), 1000 * seed + 30, "cpu").numpy().copy()
            ks = {p: synth.k_of(Lr, p) for p in SWEEP_PCTS}
            errs = {p: np.zeros_like(x) for p in SWEEP_PCTS}
            self.parts.append((Rr, Lr, x, ks, errs))
        self.input_bytes = sum(9 * 4 * Rr * Lr for Rr, Lr, _, _, _ in self.parts)  # 9 pairs
        self.sample = ("per row length, the first %s entries as rows (768, 4096, 65536) and a "
                       "whole-tensor row of %d entries; every call of the step on them"
                       % ("/".join(str(n) for _, n in ORACLE_SAMPLE[:3]), ORACLE_SAMPLE[3][1]))

    def run(self, step: int):
        o, lib = self.oracle, self.lib
        for Rr, Lr, x, ks, errs in self.parts:
            for p in SWEEP_PCTS:
                v, i = o.topk_compress(x, ks[p], lib)
                o.topk_decompress(v, i, Lr, lib)
                v, i = o.ef_topk_compress(x, errs[p], ks[p], lib)
                o.topk_decompress(v, i, Lr, lib)
            for b in SWEEP_BITS:
                c, s, m = o.quant_compress(x, b, False, 0, lib)
                o.quant_decompress(c, s, m, Lr, b, lib)


def cpu_baseline(budget_s: float = 10.0):
    st = OracleStep(0)
    st.run(0)
    n, t0 = 0, time.perf_counter()
    while time.perf_counter() - t0 < budget_s or n < 2:
        st.run(n)
        n += 1
    secs = time.perf_counter() - t0
    return {"value": round(st.input_bytes * n / secs / 1e9, 4), "unit": UNIT, "cores": 1,
            "kind": "oracle", "sample": st.sample + "; %d passes in %.1f s" % (n, secs),
            "cpu": cpu_name()}


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
        "config": {"workload": "bandwidth sweep at 2^%d entries: one N(0,1) fp32 tensor of "
                               "%d entries as rows of 768, 4096, 65536 and one whole-tensor row"
                               % (LOG2N, 1 << LOG2N),
                   "topk_percents": list(SWEEP_PCTS), "bits": list(SWEEP_BITS),
                   "oracle_sample": st.sample},
        "cpu_baseline": {"value": round(value, 4), "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": st.sample, "cpu": cpu_name()},
        "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    rank, local, world = dist_env()
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    run_headline(args, rank, local, world)
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


if __name__ == "__main__":
    main()
