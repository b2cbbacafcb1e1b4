#!/usr/bin/env python
"""Benchmark of the eviction-by-design hot path on one or more GB300s.

One step = one pass of the whole path over one batch: the eviction of every
layer through `ebd_evict` ((scoring, for the attention-scored workload) ->
select (certainty set, pi, Poisson draw, index compaction) -> gather (kept
K/V rows); the layers are independent and spread over four streams, and
within a layer the library pipelines unit chunks over its own side streams),
then the certified decode of every layer in order.  Each phase is a CUDA
graph timed between two CUDA events on the launching stream; L2 is flushed
before every phase, outside the events (a 256 MB buffer is written, then
another 256 MB buffer read, so that dirty lines are written back before the
phase starts).  The kernels of the eviction are also timed alone, one phase
each (score, select, gather), for the per-kernel rates and the roofline.

Prints ONE JSON line (rank 0).  `value` is the certified decode-step HBM
throughput in GB/s: algorithmic bytes (compact K/V rows, one log(1/pi) per
row, queries and outputs) over the decode phase's device time, summed over
ranks and divided by the slowest rank's time.

  --impl reference   times the float64 CPU oracle on a bounded sample of the
                     same workload instead (rank 0 only).
"""
from __future__ import annotations

import os

# The oracle legs are timed on one host core; set before numpy is imported.
for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, "1")

import argparse  # noqa: E402
import ctypes  # noqa: E402
import hashlib  # noqa: E402
import json  # noqa: E402
import statistics  # noqa: E402
import subprocess  # noqa: E402
import sys  # noqa: E402
import tempfile  # noqa: E402
import threading  # noqa: E402
import time  # noqa: E402

import numpy as np  # noqa: E402
import torch  # noqa: E402

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2607_21475_gb300.workloads import WORKLOADS, Workload, make_layer_inputs  # noqa: E402

METRIC = "certified decode-step HBM GB/s (% of GB300 peak) and eviction Mtokens/s"
NOMINAL_HBM_GBS = 8000.0  # the ~8 TB/s HBM3e figure quoted for GB300
FALLBACK_HBM_GBS = 6800.0
L2_FLUSH_BYTES = 256 << 20


# ----------------------------------------------------------------------------- utils
def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=50)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="dialogue_32k", choices=sorted(WORKLOADS))
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=12.0)
    p.add_argument("--no-all-cores", action="store_true",
                   help="skip the oracle timing on every host core")
    p.add_argument("--all-core-units", type=int, default=64,
                   help="units of layer 0 in the all-core oracle sample")
    p.add_argument("--no-graph", action="store_true")
    p.add_argument("--batch", type=int, default=0,
                   help="override the workload's batch (smaller cases for profiling)")
    p.add_argument("--layers", type=int, default=0,
                   help="override the workload's layer count (a smaller case of the same "
                        "kernels, e.g. for profiling)")
    p.add_argument("--sweep", action="store_true",
                   help="instead of the step: the batch x context x budget sweep on the 28/4 "
                        "GQA shape, one JSON line per point (decode GB/s and roofline "
                        "fraction, pipelined eviction Mtokens/s)")
    p.add_argument("--sweep-filter", default="",
                   help="only sweep points whose name contains this string")
    p.add_argument("--rows", action="store_true",
                   help="instead of the step: time the added rows (append/re-eviction cadence, "
                        "certificate aggregation, systematic select, observation queries, "
                        "variance contributions), one JSON line each")
    p.add_argument("--coverage", action="store_true",
                   help="instead of the step: coverage of the realised error by the "
                        "certificate over many Philox seeds, one JSON line per workload "
                        "(the Qwen-7B shape, the 16k shape at 10/25/50%%, the 32k dialogue)")
    p.add_argument("--coverage-seeds", type=int, default=200)
    return p.parse_args()


def workload_of(args) -> Workload:
    w = WORKLOADS[args.workload]
    if args.batch > 0:
        w = w.with_(batch=args.batch)
    if args.layers > 0:
        w = w.with_(n_layers=args.layers)
    return w


def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1 and args.impl == "ours":
        torch.cuda.set_device(local)
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int, device: str = "cuda") -> float:
    """The slowest rank's time: every rank's value, all-reduced with MAX."""
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x: float, world: int, device: str = "cuda") -> float:
    """Every rank's value, all-reduced with SUM (bytes of shards that differ a
    little in their kept rows)."""
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def whole_job_rate(units_per_rank: float, world: int, max_seconds: float) -> float:
    """Weak scaling: every rank processes a shard of the same size (its own B
    batch rows of the workload's shape), so the job processes world * units in
    the slowest rank's time."""
    return world * units_per_rank / max_seconds


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), "measured", pk
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback", {}


class ClockSampler:
    """SM clock and clock-event (throttle) reasons sampled during the timed region.

    Polls NVML directly (ctypes on libnvidia-ml, read-only queries) every
    millisecond from a background thread, so that even a region of a few
    milliseconds is covered; falls back to nvidia-smi at 200 ms otherwise."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, local_rank, device):
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        self.gpu = vis.split(",")[local_rank] if vis else str(local_rank)
        self.device = device
        self.samples = []
        self.reasons = 0
        self.max_mhz = None
        self.stop_flag = threading.Event()
        self.thread = None
        self.proc = None
        self.file = None
        self.nvml = None
        self.handle = None
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() != 0:
                raise OSError("nvmlInit failed")
            uuid = "GPU-" + str(torch.cuda.get_device_properties(device).uuid)
            h = ctypes.c_void_p()
            if nv.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(h)) != 0:
                raise OSError("no NVML handle")
            self.nvml, self.handle = nv, h
            mx = ctypes.c_uint()
            if nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:
                self.max_mhz = float(mx.value)
            self.reason_fn = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                getattr(nv, "nvmlDeviceGetCurrentClocksThrottleReasons")
        except (OSError, AttributeError, RuntimeError):
            self.nvml = None

    def _poll(self):
        clk = ctypes.c_uint()
        rsn = ctypes.c_ulonglong()
        while not self.stop_flag.is_set():
            if self.nvml.nvmlDeviceGetClockInfo(self.handle, 1, ctypes.byref(clk)) == 0:
                self.samples.append(float(clk.value))
            if self.reason_fn(self.handle, ctypes.byref(rsn)) == 0:
                self.reasons |= int(rsn.value)
            time.sleep(0.001)

    def start(self):
        if self.nvml is not None:
            self.thread = threading.Thread(target=self._poll, daemon=True)
            self.thread.start()
            t0 = time.time()
            while not self.samples and time.time() - t0 < 0.5:  # sampler running
                time.sleep(0.0005)
            return
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", self.gpu,
                 "--query-gpu=clocks.sm,clocks.max.sm,clocks_event_reasons.hw_slowdown,"
                 "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
                 "clocks_event_reasons.sw_power_cap", "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.file, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.thread is not None:
            self.stop_flag.set()
            self.thread.join()
            names = sorted(v for k, v in self.REASONS.items() if self.reasons & k)
            return {"sm_mhz": statistics.median(self.samples) if self.samples else None,
                    "sm_max_mhz": self.max_mhz, "reasons": names,
                    "samples": len(self.samples), "source": "nvml poll 1 ms"}
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["clock sampling unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.file.read().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 6:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[2:6]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        self.file.close()
        os.unlink(self.file.name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None, "reasons": sorted(reasons),
                "samples": len(sm), "source": "nvidia-smi 200 ms"}


def source_sha(relpath):
    with open(os.path.join(ROOT, relpath), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def traffic_for(kernel, workload):
    """DRAM bytes per launch from a committed ncu capture, if its kernel's
    sources (one file, or a list whose hashes are joined by '+') are unchanged
    since the capture (else null)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            entries = json.load(f)
    except (OSError, ValueError):
        return None
    for e in entries:
        if e.get("kernel") == kernel and e.get("workload") == workload:
            src = e["source"] if isinstance(e["source"], list) else [e["source"]]
            if e.get("source_sha") == "+".join(source_sha(f) for f in src):
                return float(e["dram_bytes_per_launch"])
    return None


# ------------------------------------------------------------------ algorithmic bytes
def decode_bytes(w: Workload, n_kept_layers):
    """Compact K/V rows + one float32 log(1/pi) per row, the queries and the outputs."""
    e = w.elem_bytes
    d = w.head_dim
    Hq = w.n_q_heads
    tot = 0
    for nk in n_kept_layers:
        tot += int(nk.sum()) * (2 * d * e + 4)
        tot += w.batch * Hq * d * e          # Q
        tot += w.batch * Hq * (d + 4) * 4    # y, lse, var, b, radius
    return tot


def gather_bytes(w: Workload, n_kept_layers):
    e, d = w.elem_bytes, w.head_dim
    return sum(int(nk.sum()) * (4 * d * e + 4) for nk in n_kept_layers)  # read + write, idx


def select_bytes(w: Workload, n_kept_layers):
    units = w.batch * w.n_kv_heads
    return sum(units * w.n_ctx * 4 + int(nk.sum()) * 8 + units * 4 for nk in n_kept_layers)


def score_flops(w: Workload):
    units = w.batch * w.n_kv_heads
    return w.n_layers * units * 2 * (2 * w.n_obs * w.group * w.n_ctx * w.head_dim)


# ------------------------------------------------------------------------- our path
class Path:
    """All device buffers of one rank's workload, plus one callable per phase."""

    def __init__(self, w: Workload, dev, use_graph: bool):
        from paper_2607_21475_gb300 import ebd
        self.ebd = ebd
        self.w = w
        self.dev = dev
        L, B, H, N, d, G = w.n_layers, w.batch, w.n_kv_heads, w.n_ctx, w.head_dim, w.group
        self.inputs = [make_layer_inputs(w, l, dev) for l in range(L)]
        self.designs = [ebd.design_for(batch=B, n_kv_heads=H, group=G, head_dim=d, n_ctx=N,
                                       layer=l, seed=w.philox_seed, n_sink=w.n_sink,
                                       n_recent=w.n_recent, k_head=w.k_head,
                                       budget_tokens=w.budget_tokens,
                                       bisect_iters=w.bisect_iters, eps=w.eps)
                        for l in range(L)]
        self.cc = [ebd.alloc_compact(B, H, w.capacity, d, w.torch_dtype, dev) for _ in range(L)]
        self.scored = w.score_kind == "attention"
        if self.scored:
            self.scores = [torch.empty((B, H, N), dtype=torch.float32, device=dev) for _ in range(L)]
            self.score_ws = torch.empty(ebd.ebd_score_workspace_bytes(B, H, w.n_obs * G),
                                        dtype=torch.uint8, device=dev)
        else:
            self.scores = [inp["scores"] for inp in self.inputs]
        Hq = w.n_q_heads
        self.out = [dict(y=torch.empty((B, Hq, d), dtype=torch.float32, device=dev),
                         **{k: torch.empty((B, Hq), dtype=torch.float32, device=dev)
                            for k in ("lse", "var", "b", "r")}) for _ in range(L)]
        dt = ebd.EBD_BF16 if w.dtype == "bf16" else ebd.EBD_F32
        self.dec_ws = torch.empty(max(1, ebd.ebd_decode_workspace_bytes(dt, B, H, G, d, w.capacity)),
                                  dtype=torch.uint8, device=dev)
        self.kernel_phases = (["score"] if self.scored else []) + ["select", "gather"]
        self.step_phases = ["evict", "decode"]
        self.phases = self.kernel_phases + self.step_phases
        # ebd_evict runs one select and one gather per chunk of SM-count units
        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        chunks = -(-(B * H) // sms)
        self.launches = {"score": 2, "select": 1, "gather": 1, "decode": 2,
                         "evict": (2 if self.scored else 0) + 2 * chunks}
        # independent layers are evicted concurrently on a few streams
        n_ev = min(L, 4) if L > 1 else 0
        self.ev_streams = [torch.cuda.Stream(device=dev) for _ in range(n_ev)]
        self.ev_ws = []
        if self.scored:
            self.ev_ws = [torch.empty(ebd.ebd_evict_workspace_bytes(self.designs[0], w.n_obs * G),
                                      dtype=torch.uint8, device=dev) for _ in range(max(1, n_ev))]
        self.use_graph = use_graph
        self.graphs = {}

    def _evict(self):
        ebd, w = self.ebd, self.w
        cur = torch.cuda.current_stream()
        streams = self.ev_streams or [cur]
        for s in self.ev_streams:
            s.wait_stream(cur)
        for l in range(w.n_layers):
            k = l % len(streams)
            inp = self.inputs[l]
            ebd.ebd_evict(self.designs[l], inp["K"], inp["V"],
                          None if self.scored else inp["scores"],
                          inp["q_obs"] if self.scored else None, self.cc[l],
                          workspace=self.ev_ws[k] if self.scored else None, stream=streams[k])
        for s in self.ev_streams:
            cur.wait_stream(s)

    # one phase over every layer
    def _run(self, phase):
        ebd, w = self.ebd, self.w
        if phase == "evict":
            return self._evict()
        for l in range(w.n_layers):
            inp, cc, o = self.inputs[l], self.cc[l], self.out[l]
            if phase == "score":
                ebd.ebd_score(inp["q_obs"], inp["K"], self.scores[l], workspace=self.score_ws)
            elif phase == "select":
                ebd.ebd_select(self.designs[l], self.scores[l], cc)
            elif phase == "gather":
                ebd.ebd_gather(self.designs[l], inp["K"], inp["V"], cc)
            else:
                ebd.ebd_certified_decode(inp["Q"], cc.K_c, cc.V_c, cc.logw_c, cc.n_kept, o["y"],
                                         o["lse"], o["var"], o["b"], o["r"],
                                         workspace=self.dec_ws)

    def capture(self):
        if not self.use_graph:
            return
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            for ph in self.phases:
                self._run(ph)
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        for ph in self.phases:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                self._run(ph)
            self.graphs[ph] = g
        torch.cuda.synchronize()

    def run(self, phase):
        if phase in self.graphs:
            self.graphs[phase].replay()
        else:
            self._run(phase)

    def status(self):
        return [int(cc.dev_status.item()) for cc in self.cc]

    def n_kept(self):
        return [torch.clamp(cc.n_kept, max=self.w.capacity).cpu().numpy() for cc in self.cc]


def e2e_run(path: Path, steps: int, in_place: bool, n_kept_layers=None):
    """Public-API end to end from page-locked host inputs, for every layer:
    ebd_evict + ebd_certified_decode, then the outputs back to host memory, all
    inside the timed region.

    in_place=False: K, V, Q and the scores (or the observation queries) are
    copied to the device first.  in_place=True: what the kernels read in full
    is copied (Q; with attention scoring also K and the observation queries,
    since scoring reads every key), the rest stays in host memory where
    ebd_evict reads it (the select reads every score, the gather only the
    kept rows).  Returns (ms per step, H2D bytes, D2H bytes), the H2D bytes
    being what crosses the link: the copies, plus for in_place the scores and
    the kept rows the kernels read in place."""
    ebd, w, dev = path.ebd, path.w, path.dev
    keys = ["K", "V", "Q"] + (["q_obs"] if path.scored else ["scores"])
    host_in = [{k: inp[k].cpu().pin_memory() for k in keys} for inp in path.inputs]
    host_out = [{k: v.cpu().pin_memory() for k, v in o.items()} for o in path.out]
    if not in_place:
        copied = keys
    elif path.scored:
        copied = ["K", "Q", "q_obs"]   # V stays on the host: only its kept rows move
    else:
        copied = ["Q"]                 # K, V and the scores stay on the host
    h2d = sum(hi[k].numel() * hi[k].element_size() for hi in host_in for k in copied)
    if in_place:
        rows = sum(int(nk.sum()) for nk in n_kept_layers)
        if path.scored:
            h2d += rows * w.head_dim * w.elem_bytes            # kept V rows
        else:
            h2d += sum(hi["scores"].numel() * 4 for hi in host_in)
            h2d += rows * 2 * w.head_dim * w.elem_bytes        # kept K and V rows
    d2h = sum(t.numel() * t.element_size() for ho in host_out for t in ho.values())
    ev_ws = None
    if path.scored:
        ev_ws = torch.empty(ebd.ebd_evict_workspace_bytes(path.designs[0], w.n_obs * w.group),
                            dtype=torch.uint8, device=dev)

    # the copies run on their own stream, layer after layer, while the
    # compute stream works on the layers already copied (each layer waits for
    # its own inputs only); a step's copies start after the previous step's
    # compute, so no input buffer is overwritten while still read
    comp = torch.cuda.current_stream()
    copy_stream = torch.cuda.Stream(device=dev)
    ready = [torch.cuda.Event() for _ in range(w.n_layers)]

    def one():
        copy_stream.wait_stream(comp)
        with torch.cuda.stream(copy_stream):
            for l in range(w.n_layers):
                for k in copied:
                    path.inputs[l][k].copy_(host_in[l][k], non_blocking=True)
                ready[l].record(copy_stream)
        for l in range(w.n_layers):
            inp, hi = path.inputs[l], host_in[l]
            comp.wait_event(ready[l])
            def src(k):
                return inp[k] if k in copied else hi[k]
            cc, o = path.cc[l], path.out[l]
            ebd.ebd_evict(path.designs[l], src("K"), src("V"),
                          None if path.scored else src("scores"),
                          inp["q_obs"] if path.scored else None, cc, workspace=ev_ws)
            ebd.ebd_certified_decode(inp["Q"], cc.K_c, cc.V_c, cc.logw_c, cc.n_kept, o["y"],
                                     o["lse"], o["var"], o["b"], o["r"], workspace=path.dec_ws)
            for k, t in o.items():
                host_out[l][k].copy_(t, non_blocking=True)

    one()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(steps):
        one()
    t1.record()
    torch.cuda.synchronize()
    return t0.elapsed_time(t1) / steps, h2d, d2h


def host_link_peak(dev, nbytes: int = 512 << 20, reps: int = 5):
    """Measured host -> device rate of this box's link: a page-locked buffer
    copied to the device (best of `reps`, CUDA events), in GB/s -- the
    denominator of the end-to-end line's link fraction."""
    src = torch.empty(nbytes, dtype=torch.uint8).pin_memory()
    dst = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    best = float("inf")
    for _ in range(reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        dst.copy_(src, non_blocking=True)
        b.record()
        torch.cuda.synchronize()
        best = min(best, a.elapsed_time(b))
    del src, dst
    return nbytes / (best * 1e-3) / 1e9


# --------------------------------------------------------------------------- oracle
def oracle_sample(w: Workload, inputs, seconds: float, max_units=None, cc=None,
                  dev_scores=None):
    """Run the float64 oracle on units of layer 0 until `seconds` of CPU time.
    Returns (units, evict_s, decode_s, decode_bytes, parity).  With `cc` (the
    device's compact cache of layer 0) each sampled unit's kept set is also
    compared with the oracle's (untimed): parity counts the tail draws with
    |u - pi| < 1e-5 (where float32 and float64 pi may decide differently),
    the units whose kept sets differ, and the differing tokens outside that
    band (0 when the path is right).  For attention-scored workloads the
    comparison evicts on the device's float32 scores (`dev_scores`)."""
    from oracle import ebd_oracle as O
    B, H, G, d = w.batch, w.n_kv_heads, w.group, w.head_dim
    units = 0
    t_ev = t_dec = 0.0
    dbytes = 0
    par = {"units": 0, "near_ties": 0, "units_differing": 0, "tokens_differing_outside_band": 0}
    if cc is not None:
        n_dev = cc.n_kept.cpu()
    total_units = B * H if max_units is None else min(max_units, B * H)
    for u in range(total_units):
        b, h = divmod(u, H)
        K = inputs["K"][b, h].double().cpu().numpy()
        V = inputs["V"][b, h].double().cpu().numpy()
        Q = inputs["Q"][b, h * G:(h + 1) * G].double().cpu().numpy()
        if w.score_kind == "attention":
            qo = inputs["q_obs"][b, h].double().cpu().numpy()
            t = time.perf_counter()
            s = O.accumulated_attention_scores(qo, K).astype(np.float32)
            t_ev += time.perf_counter() - t
        else:
            s = inputs["scores"][b, h].cpu().numpy()
        t = time.perf_counter()
        r = O.evict_unit(K, V, s, n_sink=w.n_sink, n_recent=w.n_recent, k_head=w.k_head,
                         budget_tokens=w.budget_tokens, eps=w.eps, seed=w.philox_seed, layer=0,
                         b=b, kvh=h, capacity=w.capacity)
        t_ev += time.perf_counter() - t
        t = time.perf_counter()
        O.hajek_decode(Q, r.K_c, r.V_c, r.logw)
        t_dec += time.perf_counter() - t
        n = min(r.n_kept, w.capacity)
        dbytes += n * (2 * d * w.elem_bytes + 4) + G * d * w.elem_bytes + G * (d + 4) * 4
        units += 1
        if cc is not None:
            rr = r
            if dev_scores is not None:
                rr = O.evict_unit(K, V, dev_scores[b, h].cpu().numpy(), n_sink=w.n_sink,
                                  n_recent=w.n_recent, k_head=w.k_head,
                                  budget_tokens=w.budget_tokens, eps=w.eps, seed=w.philox_seed,
                                  layer=0, b=b, kvh=h, capacity=w.capacity)
            near = ~rr.certain & (np.abs(rr.u - rr.pi) < 1e-5)
            ng = int(n_dev[b, h])
            got = set(cc.idx_c[b, h, :min(ng, w.capacity)].cpu().numpy().tolist())
            diff = got ^ set(rr.idx.tolist())
            par["units"] += 1
            par["near_ties"] += int(near.sum())
            par["units_differing"] += int(bool(diff) or ng != rr.n_kept)
            par["tokens_differing_outside_band"] += sum(1 for i in diff if not near[i])
        if t_ev + t_dec >= seconds:
            break
    return units, t_ev, t_dec, dbytes, par


def _to_f64(a):
    """float32 numpy, or bfloat16 bit patterns as int16 numpy -> float64."""
    if a.dtype == np.int16:
        return (a.astype(np.int32).astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


def _host_array(t):
    """A tensor's values for a pool worker: bf16 as its int16 bit patterns."""
    t = t.contiguous()
    return (t.view(torch.int16) if t.dtype == torch.bfloat16 else t.float()).cpu().numpy()


def _oracle_evict_task(task):
    """Pool worker: eviction of one unit (E0 first for attention scores); its
    own compute time only (the unpacking of the inputs is not timed)."""
    from oracle import ebd_oracle as O
    p, u, K16, V16, s, qo16 = task
    K, V = _to_f64(K16), _to_f64(V16)
    b, h = divmod(u, p["H"])
    t = time.perf_counter()
    if s is None:
        s = O.accumulated_attention_scores(_to_f64(qo16), K).astype(np.float32)
    r = O.evict_unit(K, V, s, n_sink=p["n_sink"], n_recent=p["n_recent"], k_head=p["k_head"],
                     budget_tokens=p["budget"], eps=p["eps"], seed=p["seed"], layer=0, b=b,
                     kvh=h, capacity=p["cap"])
    dt = time.perf_counter() - t
    return os.getpid(), dt, r.idx, r.logw


def _oracle_decode_task(task):
    """Pool worker: certified decode of one unit over its kept rows."""
    from oracle import ebd_oracle as O
    Q16, Kc16, Vc16, logw = task
    Q, Kc, Vc = _to_f64(Q16), _to_f64(Kc16), _to_f64(Vc16)
    t = time.perf_counter()
    O.hajek_decode(Q, Kc, Vc, logw)
    return os.getpid(), time.perf_counter() - t


def oracle_all_cores(w: Workload, inputs, max_units: int, processes=None):
    """The float64 oracle on every host core: a spawn-started process pool runs
    the eviction of a sample of units, then their decode; each phase's time is
    the largest per-process sum of task compute times (start-up and the
    transfer of inputs not counted)."""
    import multiprocessing as mp
    B, H, G, d = w.batch, w.n_kv_heads, w.group, w.head_dim
    cores = processes or (len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity")
                          else os.cpu_count())
    U = min(B * H, max_units)
    p = {"H": H, "n_sink": w.n_sink, "n_recent": w.n_recent, "k_head": w.k_head,
         "budget": w.budget_tokens, "eps": w.eps, "seed": w.philox_seed, "cap": w.capacity}

    i16 = _host_array
    ev_tasks = []
    for u in range(U):
        b, h = divmod(u, H)
        s = inputs["scores"][b, h].cpu().numpy() if "scores" in inputs else None
        qo = i16(inputs["q_obs"][b, h]) if s is None else None
        ev_tasks.append((p, u, i16(inputs["K"][b, h]), i16(inputs["V"][b, h]), s, qo))
    with mp.get_context("spawn").Pool(cores) as pool:
        pool.map(_to_f64, [np.zeros(1, np.int16)] * cores)  # start every worker
        res = pool.map(_oracle_evict_task, ev_tasks, chunksize=1)
        t_ev = {}
        for pid, dt, _, _ in res:
            t_ev[pid] = t_ev.get(pid, 0.0) + dt
        dec_tasks, dbytes = [], 0
        for u, (_, _, idx, logw) in enumerate(res):
            b, h = divmod(u, H)
            dec_tasks.append((i16(inputs["Q"][b, h * G:(h + 1) * G]), ev_tasks[u][2][idx],
                              ev_tasks[u][3][idx], logw))
            n = min(len(idx), w.capacity)
            dbytes += n * (2 * d * w.elem_bytes + 4) + G * d * w.elem_bytes + G * (d + 4) * 4
        t_dec = {}
        for pid, dt in pool.map(_oracle_decode_task, dec_tasks, chunksize=1):
            t_dec[pid] = t_dec.get(pid, 0.0) + dt
    wall_ev, wall_dec = max(t_ev.values()), max(t_dec.values())
    return {"value": dbytes / wall_dec / 1e9, "unit": "GB/s", "cores": cores, "kind": "oracle",
            "evict_mtok_s": U * w.n_ctx / wall_ev / 1e6,
            "sample": f"{U} of {B * H} (batch row, kv head) units of layer 0 on {cores} "
                      f"processes: eviction {wall_ev:.2f} s, decode {wall_dec:.3f} s "
                      f"(largest per-process compute time)"}


def config_of(w: Workload):
    return {"workload": w.name, "layers": w.n_layers, "batch": w.batch, "n_ctx": w.n_ctx,
            "q_heads": w.n_q_heads, "kv_heads": w.n_kv_heads, "head_dim": w.head_dim,
            "kv_dtype": w.dtype, "budget": w.budget, "budget_tokens": w.budget_tokens,
            "k_head": w.k_head, "capacity": w.capacity, "scores": w.score_kind,
            "l2": "flushed before every timed phase (256 MiB written, then 256 MiB read so "
                  "write-backs finish outside the timed region); inputs > L2"}


def run_reference(args, world, rank):
    if rank != 0:
        return
    w = workload_of(args)
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    inputs = make_layer_inputs(w, 0, dev)
    per_step = max(2.0, 150.0 / max(1, args.steps + args.warmup))
    vals, times = [], []
    units = 0
    for i in range(args.warmup + args.steps):
        t = time.perf_counter()
        u, t_ev, t_dec, db, _ = oracle_sample(w, inputs, per_step)
        dt = time.perf_counter() - t
        if i >= args.warmup:
            vals.append(db / t_dec / 1e9)
            times.append(dt * 1e3)
            units = u
    v = statistics.mean(vals)
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": "GB/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": statistics.mean(times),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_of(w),
        "cpu_baseline": {"value": v, "unit": "GB/s", "cores": 1, "kind": "oracle",
                         "sample": f"{units} of {w.batch * w.n_kv_heads} (batch row, kv head) "
                                   f"units of layer 0 per step: eviction + certified decode"},
        "e2e": {"value": v, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def run_ours(args, world, rank, local):
    w = workload_of(args)
    if rank > 0:
        # rank r holds its own shard of units: batch rows r B .. (r + 1) B - 1 of
        # a world x B batch, drawn from their own seeds (rank 0 is the
        # single-GPU workload itself)
        w = w.with_(seed=w.seed + 7919 * rank, philox_seed=w.philox_seed + rank)
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    hbm_peak, peak_kind, peaks = measured_peaks()
    path = Path(w, dev, use_graph=not args.no_graph)
    flush_w = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_r = torch.ones(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)

    def flush(i):
        # write a buffer larger than L2, then read another one: the dirty lines
        # are written back here, not inside the next timed phase
        flush_w.fill_(float(i))
        return flush_r.sum()

    for ph in path.phases:       # first eager pass (also sets kernel attributes)
        path.run(ph)
    torch.cuda.synchronize()
    path.capture()
    for _ in range(args.warmup):
        for ph in path.phases:
            flush(1)
            path.run(ph)
    torch.cuda.synchronize()
    st = path.status()
    if any(st):
        raise RuntimeError(f"device status flags raised during warm-up: {st}")
    n_kept = path.n_kept()

    ev = {ph: [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)] for ph in path.phases}
    clocks = ClockSampler(local, dev)
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    for i in range(args.steps):
        for ph in path.phases:
            flush(i)
            a, b = ev[ph][i]
            a.record()
            path.run(ph)
            b.record()
    torch.cuda.synchronize()
    barrier(world)
    clk = clocks.stop()
    ph_ms = {ph: statistics.mean(a.elapsed_time(b) for a, b in ev[ph]) for ph in path.phases}
    ph_ms = {ph: max_over_ranks(v, world) for ph, v in ph_ms.items()}
    ms_step = sum(ph_ms[p] for p in path.step_phases)

    L = w.n_layers
    dbytes = decode_bytes(w, n_kept)
    dbytes_mean = sum_over_ranks(dbytes, world) / world  # the shards' kept rows differ
    value = whole_job_rate(dbytes_mean, world, ph_ms["decode"] * 1e-3) / 1e9
    evict_mtok = whole_job_rate(w.batch * w.n_ctx * L, world, ph_ms["evict"] * 1e-3) / 1e6
    # the eviction kernels run back to back, each phase alone (no overlap)
    serial_ms = sum(ph_ms[p] for p in path.kernel_phases)
    evict_serial_mtok = whole_job_rate(w.batch * w.n_ctx * L, world, serial_ms * 1e-3) / 1e6
    kern = {
        "select": {"ms_per_launch": ph_ms["select"] / L,
                   "alg_bytes_per_launch": select_bytes(w, n_kept) / L},
        "gather": {"ms_per_launch": ph_ms["gather"] / L,
                   "alg_bytes_per_launch": gather_bytes(w, n_kept) / L},
        "decode": {"ms_per_launch": ph_ms["decode"] / L, "alg_bytes_per_launch": dbytes / L},
    }
    if path.scored:
        kern["score"] = {"ms_per_launch": ph_ms["score"] / L,
                         "alg_flops_per_launch": score_flops(w) / L}
    for k, v in kern.items():
        if "alg_bytes_per_launch" in v:
            v["gbs"] = v["alg_bytes_per_launch"] / (v["ms_per_launch"] * 1e-3) / 1e9
    dom = max(kern, key=lambda k: kern[k]["ms_per_launch"])
    kname = {"select": "evict_select_smem_kernel", "gather": "gather_rows_kernel",
             "decode": ("certified decode: decode_mma_kernel + decode_merge_kernel (split-K), "
                        "decode_cluster_kernel (few units), or decode_generic_kernel + "
                        "decode_reduce_kernel (float32 or ragged capacity), as the request "
                        "selects"),
             "score": "score_lse_tc_kernel + score_col_tc_kernel"}[dom]
    if dom == "score":
        # dense bf16 contraction on tcgen05: measured cuBLAS bf16 burst peak
        tpk = float(peaks.get("bf16_tflops", 1900.0))
        ach = kern[dom]["alg_flops_per_launch"] / (kern[dom]["ms_per_launch"] * 1e-3) / 1e12
        roof = {"bound": "tensor", "achieved": ach, "peak": tpk, "unit": "TFLOP/s",
                "frac": ach / tpk, "traffic": traffic_for(dom, w.name), "kernel": kname,
                "peak_source": f"{peak_kind} bf16 dense (MEASURED_PEAKS.json bf16_tflops)"}
    else:
        ach = kern[dom]["gbs"]
        roof = {"bound": "hbm", "achieved": ach, "peak": hbm_peak, "unit": "GB/s",
                "frac": ach / hbm_peak, "traffic": traffic_for(dom, w.name), "kernel": kname,
                "peak_source": f"{peak_kind} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)"}

    e2e = e2e_copy = None
    if not args.no_e2e:
        def e2e_line(in_place):
            ms, h2d, d2h = e2e_run(path, args.steps, in_place, n_kept)
            ms = max_over_ranks(ms, world)
            return {"value": whole_job_rate(dbytes_mean, world, ms * 1e-3) / 1e9, "unit": "GB/s",
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": ms}
        e2e_copy = e2e_line(False)
        e2e_copy["inputs"] = ("K, V, Q and the " + ("observation queries" if path.scored else
                              "scores") + " copied to the device each step")
        e2e = e2e_line(True)
        link = host_link_peak(dev)
        for line_ in (e2e, e2e_copy):
            moved = (line_["h2d_bytes_per_step"] + line_["d2h_bytes_per_step"]) / (
                line_["ms_per_step"] * 1e-3) / 1e9
            line_["host_link"] = {"achieved_gbs": moved, "h2d_peak_gbs": link,
                                  "frac": moved / link,
                                  "peak_source": "page-locked 512 MiB host->device copy, "
                                                 "best of 5, measured in this run"}
        if path.scored:
            e2e["inputs"] = ("K, Q and the observation queries copied (scoring reads every key); "
                             "V read in place from page-locked host memory (the gather reads "
                             "only the kept rows)")
        else:
            e2e["inputs"] = ("K, V and the scores read in place from page-locked host memory "
                             "(the select reads every score, the gather only the kept rows); "
                             "Q copied")

    cpu = None
    parity = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        u, t_ev, t_dec, db, par = oracle_sample(
            w, path.inputs[0], args.cpu_seconds, cc=path.cc[0],
            dev_scores=path.scores[0] if path.scored else None)
        cpu = {"value": db / t_dec / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
               "sample": f"{u} of {w.batch * w.n_kv_heads} (batch row, kv head) units of "
                         f"layer 0: eviction + certified decode ({t_ev + t_dec:.1f} s)",
               "evict_mtok_s": u * w.n_ctx / t_ev / 1e6}
        parity = dict(par, note="kept sets of the sampled layer-0 units, device against the "
                                "float64 oracle; tokens may differ only where |u - pi| < 1e-5")
        if not args.no_all_cores:
            try:
                cpu["all_cores"] = oracle_all_cores(w, path.inputs[0], args.all_core_units)
            except Exception as e:  # a host without spawn or enough memory: say so
                cpu["all_cores"] = {"unavailable": f"{type(e).__name__}: {e}"[:200]}

    launches = args.steps * sum(path.launches[p] * L for p in path.phases)
    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": w.dtype,
        "data": "synthetic (seeded torch generators; shapes of the paper's GQA decode workloads)",
        "config": config_of(w),
        "decode_pct_of_8tbs": 100.0 * value / world / NOMINAL_HBM_GBS,
        "decode_pct_of_measured_hbm": 100.0 * value / world / hbm_peak,
        "evict_mtok_s": evict_mtok, "evict_kernels_back_to_back_mtok_s": evict_serial_mtok,
        "phases_ms": ph_ms, "kernels": kern,
        "roofline": roof, "cpu_baseline": cpu, "parity_sample": parity, "e2e": e2e,
        "e2e_copy_all": e2e_copy,
        "gpu_launches": launches,
        "clocks": clk,
    }
    if rank == 0:
        print(json.dumps(line))


# ------------------------------------------------------------------ added rows
def _timer(dev, reps):
    flush_w = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    flush_r = torch.ones(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)

    def time_us(fn, n=reps):
        fn()
        torch.cuda.synchronize()
        ts = []
        for i in range(n):
            flush_w.fill_(float(i))
            flush_r.sum()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(b) * 1e3)
        return statistics.median(ts)
    return time_us


def run_rows(args):
    """One JSON line per added row, each against its bound (HBM GB/s of
    measured copy bandwidth where the row moves data, latency otherwise)."""
    from paper_2607_21475_gb300 import ebd
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    hbm_peak, peak_kind, _ = measured_peaks()
    time_us = _timer(dev, max(args.steps, 5))
    lines = []

    def emit(row, **kw):
        line = {"row": row, **kw}
        if "bytes" in kw and "us" in kw:
            gbs = kw["bytes"] / (kw["us"] * 1e-6) / 1e9
            line["gbs"] = gbs
            line["frac_of_measured_hbm"] = gbs / hbm_peak
        lines.append(line)
        print(json.dumps(line))

    def design(w, n_ctx, layer=0, seed=0, sampling=0, budget=None, k_head=None):
        return ebd.design_for(batch=w.batch, n_kv_heads=w.n_kv_heads, group=w.group,
                              head_dim=w.head_dim, n_ctx=n_ctx, layer=layer, seed=seed,
                              n_sink=w.n_sink, n_recent=w.n_recent,
                              k_head=w.k_head if k_head is None else k_head,
                              budget_tokens=w.budget_tokens if budget is None else budget,
                              bisect_iters=w.bisect_iters, eps=w.eps, sampling=sampling)

    # NEXT-1: eviction every 256 decode steps on the 16k, 25% configuration (one layer):
    # 256 x (append one token per unit + certified decode), then re-evict the grown cache
    w = WORKLOADS["qwen7b_16k_b25"].with_(n_layers=1)
    B, H, G, d, N, T = w.batch, w.n_kv_heads, w.group, w.head_dim, w.n_ctx, 256
    inp = make_layer_inputs(w, 0, dev)
    cap = w.capacity + T
    cc = ebd.alloc_compact(B, H, cap, d, w.torch_dtype, dev)
    ebd.ebd_evict(design(w, N), inp["K"], inp["V"], inp["scores"], None, cc)
    torch.cuda.synchronize()
    base = (cc.K_c.clone(), cc.V_c.clone(), cc.logw_c.clone(), cc.idx_c.clone(), cc.n_kept.clone())
    g = torch.Generator(device=dev).manual_seed(5)
    k_new = torch.randn((T, B, H, d), generator=g, device=dev).to(w.torch_dtype)
    v_new = torch.randn((T, B, H, d), generator=g, device=dev).to(w.torch_dtype)
    pos = (N + torch.arange(T, device=dev, dtype=torch.int32)).view(T, 1).expand(T, B).contiguous()
    Hq = H * G
    y = torch.empty((B, Hq, d), dtype=torch.float32, device=dev)
    o4 = [torch.empty((B, Hq), dtype=torch.float32, device=dev) for _ in range(4)]
    dec_ws = torch.empty(ebd.ebd_decode_workspace_bytes(ebd.EBD_BF16, B, H, G, d, cap),
                         dtype=torch.uint8, device=dev)

    def restore():
        for dst, src in zip((cc.K_c, cc.V_c, cc.logw_c, cc.idx_c, cc.n_kept), base):
            dst.copy_(src)

    def loop():
        for t in range(T):
            ebd.ebd_append(cc, k_new[t], v_new[t], pos[t])
            ebd.ebd_certified_decode(inp["Q"], cc.K_c, cc.V_c, cc.logw_c, cc.n_kept, y, *o4,
                                     workspace=dec_ws)
    restore()
    loop()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    restore()
    with torch.cuda.graph(graph):
        loop()
    ts = []
    for i in range(3):
        restore()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        graph.replay()
        b.record()
        torch.cuda.synchronize()
        ts.append(a.elapsed_time(b) * 1e3)
    loop_us = statistics.median(ts)
    n0 = int(base[4].sum())
    units = B * H
    e = w.elem_bytes
    dec_bytes = sum((n0 + units * (t + 1)) * (2 * d * e + 4) + B * Hq * d * e + B * Hq * (d + 4) * 4
                    for t in range(T))
    app_bytes = T * units * (2 * d * e + 8)
    assert int(cc.dev_status.item()) == 0
    # re-eviction of the grown cache (fresh seed, same budget)
    scores2 = torch.exp(torch.randn((B, H, cap), generator=g, device=dev) * 1.5)
    out = ebd.alloc_compact(B, H, cap, d, w.torch_dtype, dev)
    des2 = design(w, cap, seed=w.philox_seed + 1)
    re_us = time_us(lambda: ebd.ebd_reevict(des2, scores2, cc, out))
    kept2 = int(out.n_kept.sum())
    re_bytes = units * cap * 4 + kept2 * (4 * d * e + 16)
    emit("NEXT-1 cadence: 256 x (append + certified decode), one layer of the 16k 25% config",
         us=loop_us, bytes=dec_bytes + app_bytes, per_step_us=loop_us / T,
         workload="qwen7b_16k_b25 (B=16, 28/4 heads, d=128, N=16384), 1 layer, 256 steps")
    emit("NEXT-1 re-eviction of the grown cache (select on resident rows + row gather + compose)",
         us=re_us, bytes=re_bytes, amortized_per_step_us=re_us / T,
         workload="qwen7b_16k_b25, 1 layer, cache of N + 256 rows per unit")

    # NEXT-2: deployed certificate update, 28 layers x B=8 x 28 heads
    rad = torch.rand((28, 8, 28), device=dev)
    cert = torch.zeros(8, device=dev)
    cu_us = time_us(lambda: ebd.ebd_certificate_update(rad, cert, first_step=False))
    emit("NEXT-2 certificate update (one probed step)", us=cu_us, bytes=28 * 8 * 28 * 4 + 8 * 12,
         workload="28 layers x 8 sequences x 28 query heads")

    # NEXT-3: systematic vs Poisson select on the 32k dialogue layer
    w = WORKLOADS["dialogue_32k"]
    inp = make_layer_inputs(w, 0, dev)
    cc = ebd.alloc_compact(w.batch, w.n_kv_heads, w.capacity, w.head_dim, w.torch_dtype, dev)
    dp, ds = design(w, w.n_ctx), design(w, w.n_ctx, sampling=ebd.EBD_SAMPLING_SYSTEMATIC)
    tp = time_us(lambda: ebd.ebd_select(dp, inp["scores"], cc))
    tsy = time_us(lambda: ebd.ebd_select(ds, inp["scores"], cc))
    emit("NEXT-3 systematic select (vs Poisson select on the same scores)", us=tsy,
         poisson_us=tp, tail_sizes_exact=True,
         workload="dialogue_32k (B=32, 8 KV heads, N=32768, 10%)")

    # NEXT-4a: contributions and block scores on the dialogue compact cache
    ebd.ebd_gather(dp, inp["K"], inp["V"], ebd.ebd_select(dp, inp["scores"], cc))
    Hq = w.n_q_heads
    y = torch.empty((w.batch, Hq, w.head_dim), dtype=torch.float32, device=dev)
    o4 = [torch.empty((w.batch, Hq), dtype=torch.float32, device=dev) for _ in range(4)]
    ebd.ebd_certified_decode(inp["Q"], cc.K_c, cc.V_c, cc.logw_c, cc.n_kept, y, *o4)
    contrib = torch.empty((w.batch, Hq, w.capacity), dtype=torch.float32, device=dev)
    ct_us = time_us(lambda: ebd.ebd_variance_contributions(inp["Q"], cc.K_c, cc.V_c, cc.logw_c,
                                                           cc.n_kept, y, o4[0], contrib=contrib))
    kept = int(cc.n_kept.sum())
    ct_bytes = kept * (2 * w.head_dim * w.elem_bytes + 4) + w.batch * Hq * w.capacity * 4
    emit("NEXT-4 variance contributions (second pass over the compact cache)", us=ct_us,
         bytes=ct_bytes, workload="dialogue_32k, 256 units, 1024 query heads")
    nb = (w.n_ctx + 63) // 64
    bs_out = torch.empty((w.batch, w.n_kv_heads, nb), dtype=torch.float32, device=dev)
    bs_us = time_us(lambda: ebd.ebd_block_scores(contrib, cc.idx_c, cc.n_kept, 64, nb, out=bs_out))
    emit("NEXT-4 64-token block scores", us=bs_us, bytes=w.batch * Hq * w.capacity * 4,
         workload="dialogue_32k, 512 blocks per unit")

    # NEXT-4b: SnapKV-style window queries (last 64 prefill positions) feeding E0
    w = WORKLOADS["qwen7b_6k"]
    B, H, G, d, N = w.batch, w.n_kv_heads, w.group, w.head_dim, w.n_ctx
    Qp = torch.randn((B, H * G, N, d), generator=g, device=dev).to(torch.bfloat16)
    K = torch.randn((B, H, N, d), generator=g, device=dev).to(torch.bfloat16)
    win = torch.arange(N - 64, N, dtype=torch.int32, device=dev)
    q_obs = torch.empty((B, H, G * 64, d), dtype=torch.bfloat16, device=dev)
    gq_us = time_us(lambda: ebd.ebd_gather_queries(Qp, win, H, q_obs=q_obs))
    sc = torch.empty((B, H, N), dtype=torch.float32, device=dev)
    ws = torch.empty(ebd.ebd_score_workspace_bytes(B, H, G * 64), dtype=torch.uint8, device=dev)
    e0_us = time_us(lambda: ebd.ebd_score(q_obs, K, sc, workspace=ws))
    flops = B * H * 2 * (2 * G * 64 * N * d)
    emit("NEXT-4 SnapKV window: query gather + E0 on the window queries", us=gq_us + e0_us,
         gather_us=gq_us, e0_us=e0_us, e0_tflops=flops / (e0_us * 1e-6) / 1e12,
         workload="qwen7b_6k shape, one layer (B=8, 28/4 heads, N=6144), 64-position window")
    return lines


def run_sweep(args):
    """Batch {1,8,32,64} x N {4k,16k,64k,128k} x budget {5,10,25,50}% on the
    28/4-head, d=128, bf16 shape with log-normal scores: one layer per point,
    eviction (ebd_evict, pipelined) and certified decode each captured in a
    CUDA graph and timed alone (median of `--steps` runs, L2 flushed before
    each).  One JSON line per point."""
    from paper_2607_21475_gb300 import ebd
    from paper_2607_21475_gb300.workloads import sweep_workloads
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    hbm_peak, peak_kind, _ = measured_peaks()
    time_us = _timer(dev, max(args.steps, 5))
    for w in sweep_workloads():
        if args.sweep_filter and args.sweep_filter not in w.name:
            continue
        B, H, G, d, N = w.batch, w.n_kv_heads, w.group, w.head_dim, w.n_ctx
        inp = make_layer_inputs(w, 0, dev)
        des = ebd.design_for(batch=B, n_kv_heads=H, group=G, head_dim=d, n_ctx=N, layer=0,
                             seed=w.philox_seed, n_sink=w.n_sink, n_recent=w.n_recent,
                             k_head=w.k_head, budget_tokens=w.budget_tokens,
                             bisect_iters=w.bisect_iters, eps=w.eps)
        cc = ebd.alloc_compact(B, H, w.capacity, d, w.torch_dtype, dev)
        Hq = H * G
        y = torch.empty((B, Hq, d), dtype=torch.float32, device=dev)
        o4 = [torch.empty((B, Hq), dtype=torch.float32, device=dev) for _ in range(4)]
        ws = torch.empty(max(1, ebd.ebd_decode_workspace_bytes(ebd.EBD_BF16, B, H, G, d,
                                                               w.capacity)),
                         dtype=torch.uint8, device=dev)

        def evict():
            ebd.ebd_evict(des, inp["K"], inp["V"], inp["scores"], None, cc)

        def decode():
            ebd.ebd_certified_decode(inp["Q"], cc.K_c, cc.V_c, cc.logw_c, cc.n_kept, y, *o4,
                                     workspace=ws)

        evict()
        decode()
        torch.cuda.synchronize()
        if cc.dev_status.item():
            raise RuntimeError(f"{w.name}: device status {cc.dev_status.item()}")
        graphs = {}
        for name, fn in (("evict", evict), ("decode", decode)):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                fn()
            graphs[name] = g
        ev_us = time_us(graphs["evict"].replay)
        dec_us = time_us(graphs["decode"].replay)
        n_kept = [torch.clamp(cc.n_kept, max=w.capacity).cpu().numpy()]
        dbytes = decode_bytes(w, n_kept)
        gbs = dbytes / (dec_us * 1e-6) / 1e9
        print(json.dumps({
            "point": w.name, "batch": B, "n_ctx": N, "budget": w.budget,
            "q_heads": Hq, "kv_heads": H, "head_dim": d, "kv_dtype": w.dtype,
            "decode_us": dec_us, "decode_bytes": dbytes, "decode_gbs": gbs,
            "decode_frac_of_measured_hbm": gbs / hbm_peak, "decode_pct_of_8tbs": gbs / 80.0,
            "evict_us": ev_us, "evict_mtok_s": B * N / (ev_us * 1e-6) / 1e6,
            "peak_source": f"{peak_kind} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)"}))
        del inp, cc, y, o4, ws, graphs
        torch.cuda.empty_cache()


# ------------------------------------------------------------------ coverage
COVERAGE_WORKLOADS = ["qwen7b_6k", "qwen7b_16k_b10", "qwen7b_16k_b25", "qwen7b_16k_b50",
                      "dialogue_32k"]


def coverage_run(w: Workload, seeds, dev, layer: int = 0, delta: float = 0.1,
                 q_scale: float = 0.0):
    """Coverage of the realised error by the certificate (Section 3.4, Eq. 4):
    for each Philox seed, ebd_evict + ebd_certified_decode (both range modes)
    over the whole layer on the device, then, for every query head,
    err = ||y_hat - y|| / ||y_hat|| against the full-cache attention y of
    Eq. 1 from the float64 oracle.  Returns the fraction of (seed, head)
    cases with err <= r_t for the one-pass bound and for the exact range term,
    and medians of r_t and err.  q_scale > 0: the peaked-attention variant of
    the workload (sharpened decode queries, scores accumulated on the device
    from observation queries that resemble them; workloads.py)."""
    from oracle import ebd_oracle as O
    from paper_2607_21475_gb300 import ebd
    from paper_2607_21475_gb300.workloads import peaked_attention_inputs
    if q_scale > 0:
        inp = peaked_attention_inputs(w, layer, dev, q_scale=q_scale)
    else:
        inp = make_layer_inputs(w, layer, dev)
    B, H, G, d, N = w.batch, w.n_kv_heads, w.group, w.head_dim, w.n_ctx
    Hq = w.n_q_heads
    if "q_obs" in inp:
        scores = torch.empty((B, H, N), dtype=torch.float32, device=dev)
        ebd.ebd_score(inp["q_obs"], inp["K"], scores)
    else:
        scores = inp["scores"]
    y_full = np.empty((B, Hq, d))
    for b in range(B):
        for h in range(H):
            y_full[b, h * G:(h + 1) * G] = O.full_attention(
                inp["Q"][b, h * G:(h + 1) * G].double().cpu().numpy(),
                inp["K"][b, h].double().cpu().numpy(), inp["V"][b, h].double().cpu().numpy())
    cc = ebd.alloc_compact(B, H, w.capacity, d, w.torch_dtype, dev)
    y = torch.empty((B, Hq, d), dtype=torch.float32, device=dev)
    lse, var, bt, r_b, r_e = (torch.empty((B, Hq), dtype=torch.float32, device=dev)
                              for _ in range(5))
    errs, rbs, res = [], [], []
    for s in seeds:
        des = ebd.design_for(batch=B, n_kv_heads=H, group=G, head_dim=d, n_ctx=N, layer=layer,
                             seed=int(s), n_sink=w.n_sink, n_recent=w.n_recent, k_head=w.k_head,
                             budget_tokens=w.budget_tokens, bisect_iters=w.bisect_iters,
                             eps=w.eps)
        ebd.ebd_evict(des, inp["K"], inp["V"], scores, None, cc)
        ebd.ebd_certified_decode(inp["Q"], cc.K_c, cc.V_c, cc.logw_c, cc.n_kept, y, lse, var, bt,
                                 r_e, delta=delta, range_mode=ebd.EBD_RANGE_EXACT)
        ebd.ebd_certified_decode(inp["Q"], cc.K_c, cc.V_c, cc.logw_c, cc.n_kept, y, lse, var, bt,
                                 r_b, delta=delta, range_mode=ebd.EBD_RANGE_BOUND)
        yh = y.double().cpu().numpy()
        errs.append(np.linalg.norm(yh - y_full, axis=-1) / np.linalg.norm(yh, axis=-1))
        rbs.append(r_b.double().cpu().numpy())
        res.append(r_e.double().cpu().numpy())
    torch.cuda.synchronize()
    if cc.dev_status.item():
        raise RuntimeError(f"{w.name}: device status {cc.dev_status.item()}")
    err, rb, re_ = (np.concatenate([a.ravel() for a in x]) for x in (errs, rbs, res))
    return {
        "workload": w.name, "seeds": len(seeds), "cases": int(err.size),
        "delta": delta, "layer": layer,
        "inputs": (f"peaked: decode queries x {q_scale}, scores accumulated from observation "
                   f"queries resembling them" if q_scale > 0 else "as the workload states"),
        "coverage_bound": float(np.mean(err <= rb)), "coverage_exact": float(np.mean(err <= re_)),
        "median_radius_bound": float(np.median(rb)), "median_radius_exact": float(np.median(re_)),
        "median_rel_error": float(np.median(err)), "p99_rel_error": float(np.quantile(err, 0.99)),
        "note": ("fraction of (seed, query head) cases with ||y_hat - y|| / ||y_hat|| <= r_t, "
                 "y the full-cache attention of Eq. 1 (float64 oracle), y_hat and r_t from "
                 "the CUDA path; a reported number, not a pinned one"),
    }


def run_coverage(args):
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    names = [args.workload] if args.workload != "dialogue_32k" or "--workload" in sys.argv[1:] \
        else COVERAGE_WORKLOADS
    for name in names:
        w = WORKLOADS[name]
        for qs in (0.0, 2.0, 3.0):
            print(json.dumps(coverage_run(w, range(args.coverage_seeds), dev, q_scale=qs)))
            torch.cuda.empty_cache()


def main():
    args = parse_args()
    world, rank, local = dist_setup(args)
    if args.impl == "reference":
        run_reference(args, world, rank)
    elif args.sweep:
        if rank == 0:
            run_sweep(args)
    elif args.rows:
        if rank == 0:
            run_rows(args)
    elif args.coverage:
        if rank == 0:
            run_coverage(args)
    else:
        run_ours(args, world, rank, local)
    if world > 1 and args.impl == "ours":
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
