"""Benchmark of one GliDe-with-CaPE speculative round on the KV cache.

One step = the whole hot path for one target layer on one batch:
gamma = 5 sequential glide_cross_attn calls (draft steps), one tree_verify_attn
over the expanded proposal tree, one tree_accept.  Default workload: the
Vicuna-33B-shaped long-context case (B=4, H=52, D=128, kv_len=16384, bf16,
64-node trees), whose K/V (1.75 GB) is far larger than L2, so no flush is
needed between steps.

Prints ONE JSON line.  `value` is the KV-cache bytes the step reads
(gamma cross-attention passes + one verification pass) divided by the device
time of the step.  Beside it: every evaluation workload's round
(`per_config`), whole GliDe-with-CaPE rounds with their fixed (non-attention)
part (`cape_round`), and the calls around the round timed alone
(`next_rows`).  --impl reference times the fp64 CPU oracle instead.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import math
import multiprocessing as mp
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2402_02082_gb300 import synth  # noqa: E402

METRIC = "KV-cache HBM GB/s and fraction of ~8 TB/s peak; verified tree tokens/sec per layer"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


# ------------------------------------------------------------------ helpers
def kv_bytes(w: synth.Workload):
    """Algorithmic bytes: (cross per call, verify per call) of K/V reads only."""
    e = 2 if w.dtype == "bf16" else 4
    cross = sum(w.H * L * w.D * 2 * e for L in w.kv_len)
    verify = sum(w.H * (L + w.n) * w.D * 2 * e for L in w.kv_len)
    return cross, verify


def algo_bytes(w: synth.Workload):
    """Algorithmic bytes per launch of each kernel, inputs read + outputs written."""
    e = 2 if w.dtype == "bf16" else 4
    cross_kv, verify_kv = kv_bytes(w)
    cross = cross_kv + w.B * w.H * w.D * (e + 4) + 4 * w.B
    verify = verify_kv + w.B * w.n * w.H * w.D * (e + 4) + 4 * w.B * (w.n + 1)
    accept = w.B * w.n * (w.vocab * 4 + 4 + 4 + 4) + 8 * w.B
    return {"glide_cross_attn": cross, "tree_verify_attn": verify, "tree_accept": accept}


def measured_tflops():
    """Measured dense bf16 TFLOP/s (burst), else the fallback."""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        if "bf16_tflops" in d:
            return float(d["bf16_tflops"])
    return 1900.0


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


def kernel_source_hash(fname):
    p = os.path.join(ROOT, "paper_2402_02082_gb300", "csrc", fname)
    with open(p, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


KERNEL_FILES = {"glide_cross_attn": "cross_attn.cu", "tree_verify_attn": "tree_attn_tc.cu",
                "tree_accept": "accept.cu"}


def recorded_traffic(kernel, workload):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on
    the current source of that kernel; else None."""
    p = os.path.join(ROOT, "profiles", "dram_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    rec = d.get(kernel, {}).get(workload)
    if not rec or rec.get("source_sha256_16") != kernel_source_hash(KERNEL_FILES[kernel]):
        return None
    return rec.get("dram_bytes_per_launch")


class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.out = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, power, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
                power.append(float(parts[3]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "power_w_max": max(power) if power else None, "reasons": sorted(reasons), "samples": len(sm)}


# ----------------------------------------------------------- multi-rank
def max_over_ranks(x: float, device=None) -> float:
    """The largest value of x over all ranks (x itself without a process group).
    Timing takes the slowest rank, so a job's throughput is bounded by it."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: float, world: int, seconds: float) -> float:
    """Whole-job throughput of `world` replicas that each processed `units_per_rank`."""
    return world * units_per_rank / seconds


# ------------------------------------------------------- CPU oracle baseline
def _oracle_pair(args):
    """Oracle for one (b, h) of the step: gamma cross-attention calls + the
    tree verification (one slab of K/V)."""
    import oracle
    q_draft, q_tree, parent, Kbh, Vbh, L = args
    t0 = time.perf_counter()
    for i in range(q_draft.shape[0]):
        oracle.cross_attn(q_draft[i][None, None, None, :], Kbh[None, None], Vbh[None, None], [L])
    oracle.tree_verify_attn(q_tree[None, :, None, :], parent[None], Kbh[None, None], Vbh[None, None], [L])
    return time.perf_counter() - t0


def oracle_sample_args(w, case, pairs):
    out = []
    for b, h in pairs:
        L = w.kv_len[b]
        out.append((case["q_draft"][:, b, 0, h, :], case["q_tree"][b, :, h, :], case["parent_idx"][b],
                    np.ascontiguousarray(case["K"][b, h, :L + w.n]), np.ascontiguousarray(case["V"][b, h, :L + w.n]),
                    L))
    return out


def time_oracle(w, case, pairs, pool, cores):
    """KV GB/s of the oracle over `pairs` (b, h) slabs, with `cores` single-threaded workers."""
    args = oracle_sample_args(w, case, pairs)
    e = 2 if w.dtype == "bf16" else 4
    t0 = time.perf_counter()
    pool.map(_oracle_pair, args, chunksize=1)
    dt = time.perf_counter() - t0
    nbytes = sum(w.gamma * w.kv_len[b] * w.D * 2 * e + (w.kv_len[b] + w.n) * w.D * 2 * e for b, _ in pairs)
    return nbytes / dt / 1e9, dt


def make_pool(cores):
    os.environ["OMP_NUM_THREADS"] = "1"
    os.environ["OPENBLAS_NUM_THREADS"] = "1"
    os.environ["MKL_NUM_THREADS"] = "1"
    return mp.get_context("spawn").Pool(cores)


def pick_pairs(w, k, seed):
    g = np.random.default_rng(seed)
    allp = [(b, h) for b in range(w.B) for h in range(w.H)]
    idx = g.choice(len(allp), size=min(k, len(allp)), replace=False)
    return [allp[i] for i in sorted(idx)]


# --------------------------------------------------------------- reference
def selected_workload(args) -> synth.Workload:
    w = synth.workload(args.workload)
    if args.batch and 0 < args.batch < w.B:
        w = dataclasses.replace(w, name=f"{w.name}[:{args.batch}]", B=args.batch, kv_len=w.kv_len[:args.batch])
    return w


def run_reference(args, rank, world):
    if rank != 0:
        return 0
    w = selected_workload(args)
    case = synth.make_case(w, garbage="zero")
    cores = os.cpu_count() or 1
    pool = make_pool(cores)
    per_step = max(1, min(w.B * w.H, cores))
    for s in range(args.warmup):
        time_oracle(w, case, pick_pairs(w, per_step, 10_000 + s), pool, cores)
    total_bytes, total_t = 0.0, 0.0
    e = 2 if w.dtype == "bf16" else 4
    for s in range(args.steps):
        pairs = pick_pairs(w, per_step, s)
        gbs, dt = time_oracle(w, case, pairs, pool, cores)
        total_t += dt
        total_bytes += gbs * dt * 1e9
    pool.close()
    value = total_bytes / total_t / 1e9
    sample = (f"{per_step} of {w.B * w.H} (b,h) slabs per step: gamma={w.gamma} cross-attention calls + "
              f"tree verification each, fp64 numpy oracle, {cores} single-threaded worker processes")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total_t / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": workload_config(w),
            "cpu_baseline": {"value": value, "unit": "GB/s", "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def workload_config(w):
    return {"workload": w.name, "B": w.B, "H": w.H, "D": w.D, "kv_len": list(w.kv_len) if w.B <= 8 else "ragged",
            "tree_nodes": w.n, "gamma": w.gamma, "vocab": w.vocab, "dtype": w.dtype,
            "l2": "inputs larger than L2 (no flush)" if sum(kv_bytes(w)) > 2 * 129e6 else "L2 flushed between steps"}


# -------------------------------------------------------------------- main
# kernels each library call launches (cross-attention: the attention kernel and its merge)
LAUNCHES_PER_CALL = {"glide_cross_attn": 2, "tree_verify_attn": 1, "tree_accept": 1, "cape_expand": 1,
                     "glide_kv_compact": 1}
CAPE_MAX_TOKENS = 32   # the cap on verified tokens of the paper's CaPE runs (Section 4)
L2_BYTES = 129e6


class L2Flush:
    """Evicts the L2 (129 MB) before a timed launch by reading a 512 MB buffer:
    the L2 is left holding clean lines, so the timed kernel pays no write-back
    of the flush itself (writing the buffer instead would leave the whole L2
    dirty, and the timed kernel's own reads would then write it back)."""

    def __init__(self, dev):
        import torch
        self.buf = torch.ones(512 << 20, dtype=torch.uint8, device=dev)
        self.sink = torch.empty((), dtype=torch.int64, device=dev)

    def __call__(self):
        import torch
        torch.sum(self.buf, dim=0, dtype=torch.int64, out=self.sink)


def event_pair():
    import torch
    return torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)


class Round:
    """One workload's speculative round resident on the device, through the
    public API: gamma glide_cross_attn calls (the draft steps), one
    tree_verify_attn over the workload's tree, one tree_accept.  Also the
    pinned host copies of the per-round inputs and results for the
    end-to-end measurement."""

    def __init__(self, gb, w, dev, flags=0):
        import torch
        self.gb, self.w, self.dev, self.flags = gb, w, dev, flags
        case = synth.make_case(w, garbage="zero")
        self.case = case
        self.K, self.V = self.to_dev(case["K"]), self.to_dev(case["V"])
        self.q_draft = [self.to_dev(case["q_draft"][i]) for i in range(w.gamma)]
        self.q_tree = self.to_dev(case["q_tree"])
        self.parent = self.to_dev(case["parent_idx"].astype(np.int32))
        self.kv_len = self.to_dev(np.asarray(w.kv_len, dtype=np.int32))
        self.draft = self.to_dev(case["draft_tokens"].astype(np.int32))
        self.logits = self.to_dev(case["target_logits"])
        B, H, S_cap, D = case["K"].shape
        self.B, self.H, self.D, self.n = B, H, D, w.n
        desc = gb.make_desc(B, H, D, S_cap, gb.GLIDE_BF16 if w.dtype == "bf16" else gb.GLIDE_F32)
        self.ws = torch.zeros(gb.glide_attn_workspace_bytes(desc, w.n), dtype=torch.uint8, device=dev)
        self.ws_acc = torch.zeros(gb.glide_accept_workspace_bytes(B, w.n), dtype=torch.uint8, device=dev)
        self.out_c = [torch.empty(B, 1, H, D, device=dev) for _ in range(w.gamma)]
        self.out_t = torch.empty(B, w.n, H, D, device=dev)
        self.path = torch.empty(B, w.n, dtype=torch.int32, device=dev)
        self.ln = torch.empty(B, dtype=torch.int32, device=dev)
        self.bonus = torch.empty(B, dtype=torch.int32, device=dev)
        self.names = ["glide_cross_attn"] * w.gamma + ["tree_verify_attn", "tree_accept"]
        self._host = None

    def to_dev(self, a):
        import torch
        if a.dtype == np.uint16:
            return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(self.dev)
        return torch.from_numpy(np.ascontiguousarray(a)).to(self.dev)

    def calls(self, stream=None):
        gb, w = self.gb, self.w
        fns = [lambda i=i: gb.glide_cross_attn(self.q_draft[i], self.K, self.V, self.kv_len, w.max_kv_len,
                                               self.out_c[i], self.ws, stream=stream) for i in range(w.gamma)]
        fns.append(lambda: gb.tree_verify_attn(self.q_tree, self.parent, self.K, self.V, self.kv_len, w.max_kv_len,
                                               self.out_t, self.ws, flags=self.flags, stream=stream))
        fns.append(lambda: gb.tree_accept(self.draft, self.parent, self.logits, self.path, self.ln, self.bonus,
                                          self.ws_acc, stream=stream))
        return fns

    def step(self):
        for f in self.calls():
            f()

    def status_ok(self):
        gb = self.gb
        return gb.glide_read_device_status(self.ws) == gb.GLIDE_OK and \
            gb.glide_read_device_status(self.ws_acc) == gb.GLIDE_OK

    def kv_bytes_per_step(self):
        cross_kv, verify_kv = kv_bytes(self.w)
        return self.w.gamma * cross_kv + verify_kv

    # ---- end to end: per-round inputs from pinned host memory, results back
    def _pin_host(self):
        import torch
        w, case, n = self.w, self.case, self.w.n
        pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
        half = lambda a: a.view(np.int16) if a.dtype == np.uint16 else a
        h = {}
        h["qd"] = [pin(half(case["q_draft"][i])) for i in range(w.gamma)]
        h["qt"] = pin(half(case["q_tree"]))
        h["par"] = pin(case["parent_idx"].astype(np.int32))
        h["kv"] = pin(np.asarray(w.kv_len, dtype=np.int32))
        h["dr"] = pin(case["draft_tokens"].astype(np.int32))
        h["lg"] = pin(case["target_logits"])
        h["tk"] = [pin(half(case["K"][b, :, w.kv_len[b]:w.kv_len[b] + n])) for b in range(self.B)]
        h["tv"] = [pin(half(case["V"][b, :, w.kv_len[b]:w.kv_len[b] + n])) for b in range(self.B)]
        h["rc"] = [torch.empty(self.B, 1, self.H, self.D).pin_memory() for _ in range(w.gamma)]
        h["rt"] = torch.empty(self.B, n, self.H, self.D).pin_memory()
        h["rp"] = torch.empty(self.B, n, dtype=torch.int32).pin_memory()
        h["rl"] = torch.empty(self.B, dtype=torch.int32).pin_memory()
        h["rb"] = torch.empty(self.B, dtype=torch.int32).pin_memory()
        self._host = h

    def e2e_bytes(self):
        if self._host is None:
            self._pin_host()
        h = self._host
        nb = lambda t: t.numel() * t.element_size()
        h2d = (sum(nb(t) for t in h["qd"]) + nb(h["qt"]) + nb(h["par"]) + nb(h["kv"]) + nb(h["dr"]) + nb(h["lg"]) +
               sum(nb(t) for t in h["tk"]) + sum(nb(t) for t in h["tv"]))
        d2h = sum(nb(t) for t in h["rc"]) + nb(h["rt"]) + nb(h["rp"]) + nb(h["rl"]) + nb(h["rb"])
        return h2d, d2h

    def e2e_enqueue(self, s_comp, s_h2d, s_d2h):
        """One round through the public API with host buffers, enqueued on
        s_comp: inputs stream in on a copy stream in the order they are
        needed, each call waits only for its own inputs, and results stream
        back on a second copy stream, which s_comp joins at the end."""
        import torch
        if self._host is None:
            self._pin_host()
        h, w, n, gb = self._host, self.w, self.w.n, self.gb
        bits = lambda t: t.view(torch.int16) if t.dtype == torch.bfloat16 else t
        K16, V16 = bits(self.K), bits(self.V)
        fork = s_comp.record_event()
        s_h2d.wait_event(fork)
        s_d2h.wait_event(fork)
        ev_in = []
        with torch.cuda.stream(s_h2d):
            self.kv_len.copy_(h["kv"], non_blocking=True)
            for i in range(w.gamma):
                bits(self.q_draft[i]).copy_(h["qd"][i], non_blocking=True)
                ev_in.append(s_h2d.record_event())
            for b in range(self.B):
                K16[b, :, w.kv_len[b]:w.kv_len[b] + n].copy_(h["tk"][b], non_blocking=True)
                V16[b, :, w.kv_len[b]:w.kv_len[b] + n].copy_(h["tv"][b], non_blocking=True)
            bits(self.q_tree).copy_(h["qt"], non_blocking=True)
            self.parent.copy_(h["par"], non_blocking=True)
            ev_tree = s_h2d.record_event()
            self.draft.copy_(h["dr"], non_blocking=True)
            self.logits.copy_(h["lg"], non_blocking=True)
            ev_acc = s_h2d.record_event()

        def back(pairs):
            done = s_comp.record_event()
            s_d2h.wait_event(done)
            with torch.cuda.stream(s_d2h):
                for dst, src in pairs:
                    dst.copy_(src, non_blocking=True)

        for i in range(w.gamma):
            s_comp.wait_event(ev_in[i])
            gb.glide_cross_attn(self.q_draft[i], self.K, self.V, self.kv_len, w.max_kv_len, self.out_c[i], self.ws,
                                stream=s_comp)
            back([(h["rc"][i], self.out_c[i])])
        s_comp.wait_event(ev_tree)
        gb.tree_verify_attn(self.q_tree, self.parent, self.K, self.V, self.kv_len, w.max_kv_len, self.out_t,
                            self.ws, flags=self.flags, stream=s_comp)
        back([(h["rt"], self.out_t)])
        s_comp.wait_event(ev_acc)
        gb.tree_accept(self.draft, self.parent, self.logits, self.path, self.ln, self.bonus, self.ws_acc,
                       stream=s_comp)
        back([(h["rp"], self.path), (h["rl"], self.ln), (h["rb"], self.bonus)])
        s_comp.wait_event(s_d2h.record_event())
        s_comp.wait_event(s_h2d.record_event())


def time_e2e(enqueue, dev, steps, world):
    """Seconds for `steps` end-to-end rounds, each enqueued by enqueue(s_comp,
    s_h2d, s_d2h) and waited for: eager, and replayed as one CUDA graph (the
    host then enqueues one graph instead of every copy and launch).  Returns
    (eager_s, graph_s or None, launch description)."""
    import torch
    import torch.distributed as dist
    s_comp = torch.cuda.Stream(device=dev)   # not the legacy default stream: it can be captured
    s_h2d = torch.cuda.Stream(device=dev)
    s_d2h = torch.cuda.Stream(device=dev)

    def eager_step():
        enqueue(s_comp, s_h2d, s_d2h)
        s_comp.synchronize()

    def timed(step):
        for _ in range(2):
            step()
        if world > 1:
            dist.barrier()
        t0 = time.perf_counter()
        for _ in range(steps):
            step()
        return max_over_ranks(time.perf_counter() - t0, dev)

    eager_s = timed(eager_step)
    try:
        graph = torch.cuda.CUDAGraph()
        torch.cuda.synchronize()
        with torch.cuda.graph(graph, stream=s_comp):
            enqueue(s_comp, s_h2d, s_d2h)
        torch.cuda.synchronize()

        def graph_step():
            graph.replay()
            torch.cuda.current_stream().synchronize()
        return eager_s, timed(graph_step), "cuda_graph"
    except Exception as exc:  # capture refused on this stack: the eager round is the number
        return eager_s, None, f"eager (graph capture failed: {type(exc).__name__})"


def time_back_to_back(fns, reps, flush=None, lead_ms=4.0):
    """Average CUDA-event time (ms) of one call in a run of `reps` calls issued
    back to back on the current stream (call i is fns[i % len(fns)]), the
    way a serving loop issues them.  A GPU-side wait of about lead_ms runs
    first, so the host has enqueued every call before the first one starts:
    the run times the device, not the host's launch rate, and one event pair
    spans all the calls.  With `flush` the L2 is evicted before the run."""
    import torch
    stream = torch.cuda.current_stream()
    if flush is not None:
        flush()
    torch.cuda._sleep(int(lead_ms * 2.0e6))   # clock cycles at ~2 GHz
    a, b = event_pair()
    a.record(stream)
    for i in range(reps):
        fns[i % len(fns)]()
    b.record(stream)
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


def time_steps_events(step, steps, flush=None):
    """CUDA-event time (ms) of each of `steps` calls of step() on the current
    stream; with `flush` (an L2Flush), the L2 is evicted before every step
    (outside the timed span)."""
    import torch
    stream = torch.cuda.current_stream()
    spans = []
    for _ in range(steps):
        if flush is not None:
            flush()
        a, b = event_pair()
        a.record(stream)
        step()
        b.record(stream)
        spans.append((a, b))
    torch.cuda.synchronize()
    return [a.elapsed_time(b) for a, b in spans]


def per_config_rows(args, gb, dev, peak, head_name, head_row):
    """Every evaluation workload's round (gamma cross-attention calls, the
    verification and the acceptance), device-timed with CUDA events, and end
    to end through the public API with host buffers.  Workloads whose K/V
    fit in twice the L2 get the L2 evicted (L2Flush) before every round."""
    import torch
    rows = {}
    flush = L2Flush(dev)
    for w in synth.workloads():
        if w.name == head_name:
            rows[w.name] = head_row
            continue
        r = Round(gb, w, dev)
        for _ in range(3):
            r.step()
        torch.cuda.synchronize()
        if not r.status_ok():
            raise RuntimeError(f"device status not OK on {w.name}")
        small = sum(kv_bytes(w)) <= 2 * L2_BYTES
        fl = flush if small else None
        ms = time_steps_events(r.step, args.config_steps, fl)
        calls = {}
        for nm, f in zip(r.names, r.calls()):
            calls.setdefault(nm, []).extend(time_steps_events(f, max(3, args.config_steps // 3), fl))
        step_kv = r.kv_bytes_per_step()
        round_s = statistics.mean(ms) * 1e-3
        eager_s, graph_s, launch = time_e2e(r.e2e_enqueue, dev, args.config_steps, 1)
        e2e_s = (graph_s if graph_s is not None else eager_s) / args.config_steps
        h2d, d2h = r.e2e_bytes()
        rows[w.name] = {
            "round_us": 1e6 * round_s, "kv_bytes_per_round": step_kv, "kv_gbs": step_kv / round_s / 1e9,
            "frac_of_measured_hbm": step_kv / round_s / 1e9 / peak,
            "tree_tokens_per_s_per_layer": w.B * w.n / round_s,
            "calls_us": {k: 1e3 * statistics.mean(v) for k, v in calls.items()},
            "e2e": {"round_us": 1e6 * e2e_s, "kv_gbs": step_kv / e2e_s / 1e9, "h2d_bytes_per_round": h2d,
                    "d2h_bytes_per_round": d2h, "launch": launch},
            "l2": "evicted before every round (a 512 MB read)" if small else "K/V larger than twice L2 (no flush)",
            "shape": workload_config(w)}
        if not r.status_ok():
            raise RuntimeError(f"device status not OK on {w.name}")
        del r
        torch.cuda.empty_cache()
    del flush
    return rows


def time_cape_round(args, gb, dev, peak, name):
    """A whole GliDe-with-CaPE round on one target layer of workload `name`,
    with the tree CaPE builds: gamma glide_cross_attn calls (the draft steps),
    cape_expand over the draft's distributions (cap of 32 verified tokens, so
    33 tree nodes), tree_verify_attn over that tree, tree_accept, and
    glide_kv_compact of the accepted path.  Target logits plant the first
    four proposal tokens as argmax, so four tokens are accepted per sequence
    (the 3-4 tokens per round of the paper's CaPE runs) and compaction moves
    rows.  Device-timed (CUDA events around the round, and around the chain
    expand -> verify -> accept -> compact), L2 flushed before every round when
    the K/V fit in twice the L2; the round's fixed part is the chain less the
    verification alone.  End to end: the round's inputs from pinned host
    memory, its results back, replayed as one CUDA graph."""
    import torch
    w0 = synth.workload(name)
    n = 1 + CAPE_MAX_TOKENS
    w = dataclasses.replace(w0, name=f"{w0.name}-cape", n=n, gamma=max(w0.gamma, 5))
    B, H, D = w.B, w.H, w.D
    case = synth.make_case(w, garbage="zero")
    to = lambda a: (torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(dev)
                    if a.dtype == np.uint16 else torch.from_numpy(np.ascontiguousarray(a)).to(dev))
    K, V = to(case["K"]), to(case["V"])
    S_cap = case["K"].shape[2]
    q_draft = [to(case["q_draft"][i]) for i in range(w.gamma)]
    q_tree = to(case["q_tree"])
    kv_len = to(np.asarray(w.kv_len, dtype=np.int32))
    probs_h = synth.draft_probs(w.seed + 21, B, w.gamma, w.vocab)
    roots_h = synth.root_tokens(w.seed + 21, B, w.vocab)
    probs, roots = to(probs_h), to(roots_h)
    desc = gb.make_desc(B, H, D, S_cap, gb.GLIDE_BF16)
    ws = torch.zeros(gb.glide_attn_workspace_bytes(desc, n), dtype=torch.uint8, device=dev)
    ws_acc = torch.zeros(gb.glide_accept_workspace_bytes(B, n), dtype=torch.uint8, device=dev)
    ws_c = torch.zeros(gb.glide_cape_workspace_bytes(B, w.gamma, w.vocab), dtype=torch.uint8, device=dev)
    out_c = [torch.empty(B, 1, H, D, device=dev) for _ in range(w.gamma)]
    out_t = torch.empty(B, n, H, D, device=dev)
    tok = torch.empty(B, n, dtype=torch.int32, device=dev)
    par = torch.empty(B, n, dtype=torch.int32, device=dev)
    nn = torch.empty(B, dtype=torch.int32, device=dev)
    path = torch.empty(B, n, dtype=torch.int32, device=dev)
    ln = torch.empty(B, dtype=torch.int32, device=dev)
    bonus = torch.empty(B, dtype=torch.int32, device=dev)
    new_len = torch.empty(B, dtype=torch.int32, device=dev)
    # the tree CaPE builds (the same every round), and logits that accept its
    # first four proposal tokens
    gb.cape_expand(probs, roots, CAPE_MAX_TOKENS, tok, par, nn, ws_c)
    torch.cuda.synchronize()
    tok_h = tok.cpu().numpy()
    g = np.random.default_rng(w.seed + 22)
    lg_h = g.standard_normal((B, n, w.vocab), dtype=np.float32)
    for b in range(B):
        for i in range(1, 5):   # nodes 1..gamma are the proposal x_{t+1..t+gamma}, node i's parent is i - 1
            lg_h[b, i - 1, tok_h[b, i]] = lg_h[b, i - 1].max() + 1.0
    logits = to(lg_h)

    def expand():
        gb.cape_expand(probs, roots, CAPE_MAX_TOKENS, tok, par, nn, ws_c)

    def verify():
        gb.tree_verify_attn(q_tree, par, K, V, kv_len, w.max_kv_len, out_t, ws)

    def accept():
        gb.tree_accept(tok, par, logits, path, ln, bonus, ws_acc)

    def compact():
        gb.glide_kv_compact(K, V, kv_len, path, ln, new_len)

    def draft_steps():
        for i in range(w.gamma):
            gb.glide_cross_attn(q_draft[i], K, V, kv_len, w.max_kv_len, out_c[i], ws)

    def chain():
        expand()
        verify()
        accept()
        compact()

    def whole():
        draft_steps()
        chain()

    for _ in range(3):
        whole()
    torch.cuda.synchronize()
    accepted = [int(x) for x in ln.cpu().tolist()]
    small = sum(kv_bytes(w)) <= 2 * L2_BYTES
    flush = L2Flush(dev) if small else None
    steps = args.config_steps
    t_round = statistics.mean(time_steps_events(whole, steps, flush))
    t_chain = statistics.mean(time_steps_events(chain, steps, flush))
    t_verify = statistics.mean(time_steps_events(verify, steps, flush))
    t_draft = statistics.mean(time_steps_events(draft_steps, steps, flush))
    for wsx in (ws, ws_acc, ws_c):
        if gb.glide_read_device_status(wsx) != gb.GLIDE_OK:
            raise RuntimeError("device status not OK in the CaPE round")

    # end to end: the draft queries, draft distributions, roots, tree queries,
    # the tree's own K/V rows, kv_len and the target logits come from pinned
    # host memory; the attention outputs, the accepted path and the new
    # lengths go back
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
    half = lambda a: a.view(np.int16) if a.dtype == np.uint16 else a
    h_qd = [pin(half(case["q_draft"][i])) for i in range(w.gamma)]
    h_qt, h_pr, h_rt = pin(half(case["q_tree"])), pin(probs_h), pin(roots_h)
    h_kv, h_lg = pin(np.asarray(w.kv_len, dtype=np.int32)), pin(lg_h)
    h_tk = [pin(half(case["K"][b, :, w.kv_len[b]:w.kv_len[b] + n])) for b in range(B)]
    h_tv = [pin(half(case["V"][b, :, w.kv_len[b]:w.kv_len[b] + n])) for b in range(B)]
    r_c = [torch.empty(B, 1, H, D).pin_memory() for _ in range(w.gamma)]
    r_t = torch.empty(B, n, H, D).pin_memory()
    r_p = torch.empty(B, n, dtype=torch.int32).pin_memory()
    r_l, r_b, r_n = (torch.empty(B, dtype=torch.int32).pin_memory() for _ in range(3))
    bits = lambda t: t.view(torch.int16) if t.dtype == torch.bfloat16 else t
    K16, V16 = bits(K), bits(V)

    def enqueue(s_comp, s_h2d, s_d2h):
        fork = s_comp.record_event()
        s_h2d.wait_event(fork)
        s_d2h.wait_event(fork)
        ev = []
        with torch.cuda.stream(s_h2d):
            kv_len.copy_(h_kv, non_blocking=True)
            for i in range(w.gamma):
                bits(q_draft[i]).copy_(h_qd[i], non_blocking=True)
                ev.append(s_h2d.record_event())
            probs.copy_(h_pr, non_blocking=True)
            roots.copy_(h_rt, non_blocking=True)
            ev_exp = s_h2d.record_event()
            for b in range(B):
                K16[b, :, w.kv_len[b]:w.kv_len[b] + n].copy_(h_tk[b], non_blocking=True)
                V16[b, :, w.kv_len[b]:w.kv_len[b] + n].copy_(h_tv[b], non_blocking=True)
            bits(q_tree).copy_(h_qt, non_blocking=True)
            ev_tree = s_h2d.record_event()
            logits.copy_(h_lg, non_blocking=True)
            ev_acc = s_h2d.record_event()

        def back(pairs):
            done = s_comp.record_event()
            s_d2h.wait_event(done)
            with torch.cuda.stream(s_d2h):
                for dst, src in pairs:
                    dst.copy_(src, non_blocking=True)

        with torch.cuda.stream(s_comp):
            for i in range(w.gamma):
                s_comp.wait_event(ev[i])
                gb.glide_cross_attn(q_draft[i], K, V, kv_len, w.max_kv_len, out_c[i], ws, stream=s_comp)
                back([(r_c[i], out_c[i])])
            s_comp.wait_event(ev_exp)
            gb.cape_expand(probs, roots, CAPE_MAX_TOKENS, tok, par, nn, ws_c, stream=s_comp)
            s_comp.wait_event(ev_tree)
            gb.tree_verify_attn(q_tree, par, K, V, kv_len, w.max_kv_len, out_t, ws, stream=s_comp)
            back([(r_t, out_t)])
            s_comp.wait_event(ev_acc)
            gb.tree_accept(tok, par, logits, path, ln, bonus, ws_acc, stream=s_comp)
            gb.glide_kv_compact(K, V, kv_len, path, ln, new_len, stream=s_comp)
            back([(r_p, path), (r_l, ln), (r_b, bonus), (r_n, new_len)])
        s_comp.wait_event(s_d2h.record_event())
        s_comp.wait_event(s_h2d.record_event())

    eager_s, graph_s, launch = time_e2e(enqueue, dev, steps, 1)
    e2e_us = 1e6 * (graph_s if graph_s is not None else eager_s) / steps
    nb = lambda t: t.numel() * t.element_size()
    h2d = (sum(nb(t) for t in h_qd) + nb(h_qt) + nb(h_pr) + nb(h_rt) + nb(h_kv) + nb(h_lg) +
           sum(nb(t) for t in h_tk) + sum(nb(t) for t in h_tv))
    d2h = sum(nb(t) for t in r_c) + nb(r_t) + nb(r_p) + 3 * nb(r_l)
    step_kv = sum(kv_bytes(w)[0] for _ in range(w.gamma)) + kv_bytes(w)[1]
    del K, V, flush
    torch.cuda.empty_cache()
    return {"round_us": 1e3 * t_round, "draft_steps_us": 1e3 * t_draft, "chain_us": 1e3 * t_chain,
            "verify_us": 1e3 * t_verify, "fixed_us": 1e3 * (t_chain - t_verify),
            "kv_gbs": step_kv / (t_round * 1e-3) / 1e9, "frac_of_measured_hbm": step_kv / (t_round * 1e-3) / 1e9 / peak,
            "accepted": accepted, "tree_nodes": n,
            "e2e": {"round_us": e2e_us, "kv_gbs": step_kv / (e2e_us * 1e-6) / 1e9, "h2d_bytes_per_round": h2d,
                    "d2h_bytes_per_round": d2h, "launch": launch},
            "l2": "evicted before every round (a 512 MB read)" if small else "K/V larger than twice L2 (no flush)",
            "shape": f"B={B} H={H} D={D} kv_len={list(w.kv_len)} gamma={w.gamma} V={w.vocab}, "
                     f"CaPE tree of {n} nodes (cap {CAPE_MAX_TOKENS}), one layer"}


def time_next_rows(args, w, case, gb, dev, stream, K, V, kv_len, peak):
    """CaPE expansion of this workload's gamma draft distributions over the
    Vicuna vocabulary, and the cache update of one accepted path per tree,
    each launched `args.next_iters` times with the L2 evicted (L2Flush) before
    every launch; CUDA-event time of the launch alone."""
    import torch
    iters = max(3, args.next_iters)
    flush = L2Flush(dev)

    def timed(fn):
        ms = time_steps_events(fn, iters + 2, flush)[2:]
        return sum(ms) / len(ms)

    B = w.B
    probs = torch.from_numpy(synth.draft_probs(w.seed + 17, B, w.gamma, w.vocab)).to(dev)
    roots = torch.from_numpy(synth.root_tokens(w.seed + 17, B, w.vocab)).to(dev)
    n_out = 1 + CAPE_MAX_TOKENS
    tok = torch.empty(B, n_out, dtype=torch.int32, device=dev)
    par = torch.empty(B, n_out, dtype=torch.int32, device=dev)
    nn = torch.empty(B, dtype=torch.int32, device=dev)
    conf = torch.empty(B, w.gamma, device=dev)
    ws_c = torch.zeros(gb.glide_cape_workspace_bytes(B, w.gamma, w.vocab), dtype=torch.uint8, device=dev)
    cape_ms = timed(lambda: gb.cape_expand(probs, roots, CAPE_MAX_TOKENS, tok, par, nn, ws_c, conf=conf))
    cape_bytes = probs.numel() * 4 + B * 4 + 2 * B * n_out * 4 + B * 4 + B * w.gamma * 4
    nodes = nn.cpu().tolist()

    # Accepted paths for the cache update: the step's own acceptance on random
    # logits accepts almost nothing, so take, in each tree, the root path to the
    # highest-numbered node of depth min(4, tree depth): an accepted length
    # like the 3-4 tokens per round of the paper's CaPE runs, with every
    # accepted entry moving.
    par_h = case["parent_idx"]
    n = par_h.shape[1]
    p_h = np.full((B, n), -1, dtype=np.int32)
    l_h = np.zeros(B, dtype=np.int32)
    for b in range(B):
        depth = synth.tree_depths(par_h[b])
        d = min(4, int(depth.max()))
        c = max(i for i in range(n) if depth[i] == d)
        chain = [c]
        while chain[-1] != 0:
            chain.append(int(par_h[b, chain[-1]]))
        p_h[b, :len(chain)] = chain[::-1]
        l_h[b] = len(chain) - 1
    path_c = torch.from_numpy(p_h).to(dev)
    len_c = torch.from_numpy(l_h).to(dev)
    new_len = torch.empty(B, dtype=torch.int32, device=dev)
    comp_ms = timed(lambda: gb.glide_kv_compact(K, V, kv_len, path_c, len_c, new_len))
    e = 2 if w.dtype == "bf16" else 4
    moved = sum(1 for b in range(B) for k in range(1, int(l_h[b]) + 1) if int(p_h[b, k]) != k)
    comp_bytes = moved * w.H * w.D * e * 2 * 2 + B * (4 * 3 + 4 * (int(l_h.max()) + 1))
    # speculative-sampling acceptance of a gamma-token chain (the GliDe-alone setting)
    sq = synth.draft_probs(w.seed + 18, B, w.gamma, w.vocab)
    s_draft = torch.from_numpy(synth.sample_tokens(w.seed + 18, sq)).to(dev)
    s_logits = torch.from_numpy(synth.target_logits_near(w.seed + 18, sq, 0.7)).to(dev)
    s_u = torch.from_numpy(synth.uniforms(w.seed + 18, (B, w.gamma + 1))).to(dev)
    s_q = torch.from_numpy(sq).to(dev)
    s_n = torch.empty(B, dtype=torch.int32, device=dev)
    s_t = torch.empty(B, dtype=torch.int32, device=dev)
    ws_s = torch.zeros(gb.glide_sample_workspace_bytes(B, w.gamma), dtype=torch.uint8, device=dev)
    samp_ms = timed(lambda: gb.spec_sample_accept(s_draft, s_q, s_logits, s_u, s_n, s_t, ws_s))
    # logits once, one draft row for the residual draw, the draft tokens' probabilities
    samp_bytes = B * (w.gamma + 1) * w.vocab * 4 + B * w.vocab * 4 + B * w.gamma * 8 + B * (w.gamma + 1) * 4 + 8 * B
    # grouped-query attention on the Mistral-7B shape (32 query heads over 8
    # cached heads, D = 128), this workload's batch and context, the gamma = 5
    # chain of GliDe alone: one cross-attention call and one verification
    Hq, Hk, n6 = 32, 8, w.gamma + 1
    n33 = 1 + CAPE_MAX_TOKENS   # a CaPE-sized tree: 132 query rows per cached head
    Lk = max(w.kv_len)
    Sg = (Lk + n33 + 15) // 16 * 16
    gK = torch.randn(B, Hk, Sg, w.D, device=dev, dtype=torch.bfloat16)
    gV = torch.randn_like(gK)
    g_kv = torch.full((B,), Lk, dtype=torch.int32, device=dev)
    g_qd = torch.randn(B, 1, Hq, w.D, device=dev, dtype=torch.bfloat16)
    g_qt = torch.randn(B, n6, Hq, w.D, device=dev, dtype=torch.bfloat16)
    g_par = torch.arange(-1, n6 - 1, dtype=torch.int32, device=dev).repeat(B, 1).contiguous()
    g_oc = torch.empty(B, 1, Hq, w.D, device=dev)
    g_ot = torch.empty(B, n6, Hq, w.D, device=dev)
    g_ws = torch.zeros(gb.glide_attn_workspace_bytes(gb.make_desc(B, Hq, w.D, Sg, gb.GLIDE_BF16, H_kv=Hk), n33),
                       dtype=torch.uint8, device=dev)
    gqa_c_ms = timed(lambda: gb.glide_cross_attn(g_qd, gK, gV, g_kv, Lk, g_oc, g_ws))
    gqa_t_ms = timed(lambda: gb.tree_verify_attn(g_qt, g_par, gK, gV, g_kv, Lk, g_ot, g_ws))
    g_qt33 = torch.randn(B, n33, Hq, w.D, device=dev, dtype=torch.bfloat16)
    g_par33 = torch.from_numpy(np.stack([synth.random_tree(w.seed + 40 + b, n33, 6, 5) for b in range(B)])).to(dev)
    g_ot33 = torch.empty(B, n33, Hq, w.D, device=dev)
    gqa_t33_ms = timed(lambda: gb.tree_verify_attn(g_qt33, g_par33, gK, gV, g_kv, Lk, g_ot33, g_ws))
    gqa_t33_bytes = B * Hk * (Lk + n33) * w.D * 2 * 2 + B * n33 * Hq * w.D * (2 + 4) + 4 * B * (n33 + 1)
    gqa_c_bytes = B * Hk * Lk * w.D * 2 * 2 + B * Hq * w.D * (2 + 4)
    gqa_t_bytes = B * Hk * (Lk + n6) * w.D * 2 * 2 + B * n6 * Hq * w.D * (2 + 4) + 4 * B * (n6 + 1)
    # the same calls over the caches of eight layers in turn, back to back, as
    # a verification pass over a target model's layers issues them (each
    # layer's cache is its own, so every call reads its K/V from HBM)
    n_lay = 8
    lay = [(gK, gV)] + [(torch.randn_like(gK), torch.randn_like(gV)) for _ in range(n_lay - 1)]
    gqa_layers = {}
    for nm, mk, nb in (("cross", lambda k, v: lambda: gb.glide_cross_attn(g_qd, k, v, g_kv, Lk, g_oc, g_ws), gqa_c_bytes),
                       ("verify", lambda k, v: lambda: gb.tree_verify_attn(g_qt, g_par, k, v, g_kv, Lk, g_ot, g_ws),
                        gqa_t_bytes),
                       ("verify_cape", lambda k, v: lambda: gb.tree_verify_attn(g_qt33, g_par33, k, v, g_kv, Lk, g_ot33,
                                                                                g_ws), gqa_t33_bytes)):
        fns = [mk(k, v) for k, v in lay]
        ms = statistics.median(time_back_to_back(fns, 4 * n_lay) for _ in range(3))
        gqa_layers[nm + "_us"] = 1e3 * ms
        gqa_layers[nm + "_gbs"] = nb / (ms * 1e-3) / 1e9
        gqa_layers[nm + "_frac_of_peak"] = nb / (ms * 1e-3) / 1e9 / peak
    gqa_layers["how"] = (f"{n_lay} layers' caches in turn, {4 * n_lay} calls back to back, one event pair "
                         "around the run (mean call duration)")
    del lay, gK, gV
    # the draft's training-time cross-attention under the block mask (L = 5) on a
    # Vicuna-7B training shape: B = 4 sequences of T = 2048, 32 heads, D = 128
    Bt, Tt, Ht, Lb = 4, 2048, 32, 5
    tK = torch.randn(Bt, Ht, Tt, w.D, device=dev, dtype=torch.bfloat16)
    tV = torch.randn_like(tK)
    tq = torch.randn(Bt, Tt, Ht, w.D, device=dev, dtype=torch.bfloat16)
    t_out = torch.empty(Bt, Tt, Ht, w.D, device=dev)
    t_len = torch.full((Bt,), Tt, dtype=torch.int32, device=dev)
    t_ws = torch.zeros(gb.glide_block_attn_workspace_bytes(gb.make_desc(Bt, Ht, w.D, Tt, gb.GLIDE_BF16), Tt),
                       dtype=torch.uint8, device=dev)
    blk_ms = timed(lambda: gb.glide_block_cross_attn(tq, tK, tV, t_len, Lb, t_out, t_ws))
    vis = sum(Lb * (j // Lb) for j in range(Tt))             # visible (query, key) pairs per (b, h)
    blk_flops = 4.0 * w.D * vis * Bt * Ht                    # two products, 2 flops per multiply-add
    blk_bytes = 2 * tK.numel() * 2 + tq.numel() * 2 + t_out.numel() * 4
    tf_peak = measured_tflops()
    del tK, tV, tq, t_out, t_ws
    del flush
    return {
        "block_mask_training_shape": {
            "avg_us": 1e3 * blk_ms, "tflops": blk_flops / (blk_ms * 1e-3) / 1e12,
            "frac_of_bf16_peak": blk_flops / (blk_ms * 1e-3) / 1e12 / tf_peak,
            "gbs_of_compulsory_bytes": blk_bytes / (blk_ms * 1e-3) / 1e9,
            "shape": f"B={Bt} T={Tt} H={Ht} D={w.D} L={Lb} bf16 (Vicuna-7B training shape)"},
        "gqa_mistral7b_shape": {
            "cross_us": 1e3 * gqa_c_ms, "cross_gbs": gqa_c_bytes / (gqa_c_ms * 1e-3) / 1e9,
            "cross_frac_of_peak": gqa_c_bytes / (gqa_c_ms * 1e-3) / 1e9 / peak,
            "verify_us": 1e3 * gqa_t_ms, "verify_gbs": gqa_t_bytes / (gqa_t_ms * 1e-3) / 1e9,
            "verify_frac_of_peak": gqa_t_bytes / (gqa_t_ms * 1e-3) / 1e9 / peak,
            "verify_cape_us": 1e3 * gqa_t33_ms, "verify_cape_gbs": gqa_t33_bytes / (gqa_t33_ms * 1e-3) / 1e9,
            "verify_cape_frac_of_peak": gqa_t33_bytes / (gqa_t33_ms * 1e-3) / 1e9 / peak,
            "layers_back_to_back": gqa_layers,
            "shape": f"B={B} H=32 over H_kv=8 D={w.D} kv_len={Lk} bf16, chain of {n6} nodes; "
                     f"verify_cape: a random {n33}-node tree (CaPE's 32 verified tokens and the root)"},
        "spec_sample_accept": {"avg_us": 1e3 * samp_ms, "algo_bytes_per_launch": samp_bytes,
                               "achieved_gbs": samp_bytes / (samp_ms * 1e-3) / 1e9,
                               "frac_of_peak": samp_bytes / (samp_ms * 1e-3) / 1e9 / peak,
                               "accepted": [int(x) for x in s_n.cpu().tolist()],
                               "shape": f"B={B} gamma={w.gamma} V={w.vocab} fp32 chain"},
        "cape_expand": {"avg_us": 1e3 * cape_ms, "algo_bytes_per_launch": cape_bytes,
                        "achieved_gbs": cape_bytes / (cape_ms * 1e-3) / 1e9,
                        "frac_of_peak": cape_bytes / (cape_ms * 1e-3) / 1e9 / peak,
                        "shape": f"B={B} gamma={w.gamma} V={w.vocab} fp32, cap {CAPE_MAX_TOKENS}",
                        "tree_nodes": nodes},
        "glide_kv_compact": {"avg_us": 1e3 * comp_ms, "algo_bytes_per_launch": comp_bytes,
                             "achieved_gbs": comp_bytes / (comp_ms * 1e-3) / 1e9,
                             "frac_of_peak": comp_bytes / (comp_ms * 1e-3) / 1e9 / peak,
                             "moved_rows": moved, "accepted_len": [int(x) for x in l_h],
                             "shape": f"one layer, B={B} H={w.H} D={w.D} {w.dtype}"},
        "iters": iters, "l2": "evicted before every launch (a 512 MB read)",
    }


def run_glide(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist

    from paper_2402_02082_gb300 import binding as gb
    from paper_2402_02082_gb300 import build

    if rank == 0 or world == 1:
        build.build()
    if world > 1:
        dist.barrier()
    build.build()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w = selected_workload(args)

    cpu = None
    if world == 1 and rank == 0 and not args.no_cpu_baseline:
        cores = os.cpu_count() or 1
        pool = make_pool(cores)   # spawned before any GPU work
        cpu = (pool, cores)

    r = Round(gb, w, dev, gb.GLIDE_FLAG_FORCE_FMA if args.force_fma else 0)
    B, H, n = r.B, r.H, r.n
    step_fns = r.calls()
    names = r.names
    stream = torch.cuda.current_stream()

    for _ in range(args.warmup):
        r.step()
    torch.cuda.synchronize()
    if not r.status_ok():
        raise RuntimeError("device status not OK after warm-up")

    # ---- device-timed region: inputs resident in HBM.  The step's calls run
    # back to back, as in a serving loop (one event pair around the region:
    # events between the calls would add their own cost and break the
    # programmatic launch chain from one call to the next).
    t_begin, t_end = event_pair()
    clocks = ClockSampler(local_rank)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    t_begin.record(stream)
    for s in range(args.steps):
        for f in step_fns:
            f()
    t_end.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    if world > 1:
        dist.barrier()
    elapsed_ms = t_begin.elapsed_time(t_end)
    elapsed_ms = max_over_ranks(elapsed_ms, dev)
    if not r.status_ok():
        raise RuntimeError("device status not OK after the timed region")

    # ---- the same steps again with an event pair around every call, for the
    # per-kernel durations (roofline) and shares
    ev = [[event_pair() for _ in step_fns] for _ in range(args.steps)]
    torch.cuda.synchronize()
    for s in range(args.steps):
        for j, f in enumerate(step_fns):
            ev[s][j][0].record(stream)
            f()
            ev[s][j][1].record(stream)
    torch.cuda.synchronize()
    per_kernel = {}
    for j, nm in enumerate(names):
        per_kernel.setdefault(nm, []).extend(ev[s][j][0].elapsed_time(ev[s][j][1]) for s in range(args.steps))
    if not r.status_ok():
        raise RuntimeError("device status not OK after the per-call timing")

    # ---- each call back to back (the per-call durations of the roofline and
    # the shares): events around a single short launch also time the event
    # machinery (~2 us steps on this GPU) and the launch itself.  The K/V
    # caches are far larger than L2; the logits rows of tree_accept are not,
    # so its calls rotate over enough copies of them (> 2 x L2) that every
    # call reads its logits from HBM.
    import torch
    g = w.gamma
    n_acc = max(2, int(math.ceil(2 * L2_BYTES / max(1, r.logits.numel() * 4))))
    acc_logits = [r.logits] + [r.logits.clone() for _ in range(n_acc - 1)]
    acc_fns = [lambda lg=lg: gb.tree_accept(r.draft, r.parent, lg, r.path, r.ln, r.bonus, r.ws_acc)
               for lg in acc_logits]
    b2b_ms = {}
    for nm, fns, reps in (("glide_cross_attn", step_fns[:g], 2 * g), ("tree_verify_attn", step_fns[g:g + 1], 8),
                          ("tree_accept", acc_fns, 64)):
        b2b_ms[nm] = statistics.median(time_back_to_back(fns, reps) for _ in range(3))
    del acc_logits, acc_fns
    if not r.status_ok():
        raise RuntimeError("device status not OK after the back-to-back timing")

    step_kv = r.kv_bytes_per_step()
    value = job_throughput(step_kv * args.steps, world, elapsed_ms * 1e-3) / 1e9
    tree_tok = job_throughput(B * n * args.steps, world, elapsed_ms * 1e-3)

    # ---- the acceptance's cost inside the round: [verify, accept] minus [verify]
    # back to back (events around a single short launch also time the event
    # machinery, ~2 us steps on this GPU, and break the programmatic launch
    # chain between the two calls)
    pairs_va, pairs_v = [], []
    for _ in range(max(10, args.steps // 4)):
        for lst, fns in ((pairs_va, step_fns[-2:]), (pairs_v, step_fns[-2:-1])):
            a, b = event_pair()
            a.record(stream)
            for f in fns:
                f()
            b.record(stream)
            lst.append((a, b))
    torch.cuda.synchronize()
    accept_marginal_ms = (statistics.mean(a.elapsed_time(b) for a, b in pairs_va) -
                          statistics.mean(a.elapsed_time(b) for a, b in pairs_v))

    # ---- end to end: per-round inputs from pinned host memory, results back to host
    e2e_steps = max(3, min(args.steps, args.e2e_steps))
    e2e_eager_s, e2e_graph_s, e2e_launch = time_e2e(r.e2e_enqueue, dev, e2e_steps, world)
    e2e_s = e2e_graph_s if e2e_graph_s is not None else e2e_eager_s
    e2e_value = job_throughput(step_kv * e2e_steps, world, e2e_s) / 1e9
    e2e_eager = job_throughput(step_kv * e2e_steps, world, e2e_eager_s) / 1e9
    h2d, d2h = r.e2e_bytes()

    # ---- the calls around the round (each timed alone with L2 flushed), every
    # evaluation workload's round, and whole CaPE rounds
    peak, peak_src = measured_peaks()
    next_rows = time_next_rows(args, w, r.case, gb, dev, stream, r.K, r.V, r.kv_len, peak)

    # ---- roofline of the dominant kernel
    ab = algo_bytes(w)
    kernels = {}
    tot_ms = sum(names.count(k) * v for k, v in b2b_ms.items())
    for nm, times in per_kernel.items():
        avg_ms = b2b_ms[nm]
        ach = ab[nm] / (avg_ms * 1e-3) / 1e9
        kernels[nm] = {"avg_us": 1e3 * avg_ms, "launches_per_step": names.count(nm),
                       "share": names.count(nm) * avg_ms / tot_ms,
                       "algo_bytes_per_launch": ab[nm], "achieved_gbs": ach, "frac_of_peak": ach / peak,
                       "how": "mean call duration in a run of back-to-back calls, one event pair around the run",
                       "alone_us": 1e3 * sum(times) / len(times)}
    acc_b = ab["tree_accept"]
    kernels["tree_accept"]["in_round"] = {
        "marginal_us": 1e3 * accept_marginal_ms, "achieved_gbs": acc_b / (accept_marginal_ms * 1e-3) / 1e9,
        "frac_of_peak": acc_b / (accept_marginal_ms * 1e-3) / 1e9 / peak,
        "how": "mean of [tree_verify_attn, tree_accept] minus mean of [tree_verify_attn], back to back"}
    dom = max(kernels, key=lambda k: kernels[k]["share"])
    roof = {"kernel": dom, "bound": "hbm", "achieved": kernels[dom]["achieved_gbs"], "peak": peak,
            "peak_source": peak_src, "unit": "GB/s", "frac": kernels[dom]["frac_of_peak"],
            "traffic": recorded_traffic(dom, w.name)}

    per_config, cape_round = None, None
    if world == 1 and not args.no_per_config:
        round_s = elapsed_ms * 1e-3 / args.steps
        head = {"round_us": 1e6 * round_s, "kv_bytes_per_round": step_kv, "kv_gbs": step_kv / round_s / 1e9,
                "frac_of_measured_hbm": step_kv / round_s / 1e9 / peak,
                "tree_tokens_per_s_per_layer": B * n / round_s,
                "calls_us": {k: v["avg_us"] for k, v in kernels.items()},
                "e2e": {"round_us": 1e6 * e2e_s / e2e_steps, "kv_gbs": step_kv / (e2e_s / e2e_steps) / 1e9,
                        "h2d_bytes_per_round": h2d, "d2h_bytes_per_round": d2h, "launch": e2e_launch},
                "l2": "K/V larger than twice L2 (no flush)", "shape": workload_config(w),
                "note": "the headline measurement above"}
        per_config = per_config_rows(args, gb, dev, peak, w.name, head)
        cape_round = {nm: time_cape_round(args, gb, dev, peak, nm)
                      for nm in dict.fromkeys(("vicuna7b-chain", args.workload))}

    cpu_baseline = None
    if cpu is not None:
        pool, cores = cpu
        pairs = pick_pairs(w, args.cpu_pairs or w.B * w.H, 1234)
        gbs, dt = time_oracle(w, r.case, pairs, pool, cores)
        pool.close()
        cpu_baseline = {"value": gbs, "unit": "GB/s", "cores": cores, "kind": "oracle",
                        "sample": f"{len(pairs)} of {B * H} (b,h) slabs: gamma={w.gamma} cross-attention calls + "
                                  f"tree verification each; fp64 numpy oracle, {cores} single-threaded workers, "
                                  f"{dt:.1f} s wall"}

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": elapsed_ms / args.steps, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
                "config": workload_config(w),
                "frac_of_nominal_8tbs": value / world / NOMINAL_HBM_GBS,
                "frac_of_measured_hbm": value / world / peak,
                "tree_tokens_per_s_per_layer": tree_tok,
                "roofline": roof, "kernels": kernels, "per_config": per_config, "cape_round": cape_round,
                "next_rows": next_rows, "cpu_baseline": cpu_baseline,
                "e2e": {"value": e2e_value, "unit": "GB/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                        "steps": e2e_steps, "launch": e2e_launch, "eager_value": e2e_eager},
                "gpu_launches": sum(LAUNCHES_PER_CALL[nm] for nm in names) * args.steps, "clocks": clk}
        if args.force_fma:
            line["config"]["tree_kernel"] = "cuda-core (forced)"
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["glide", "reference"], default="glide")
    ap.add_argument("--workload", default="vicuna33b-long-b4", choices=[w.name for w in synth.workloads()])
    ap.add_argument("--e2e-steps", type=int, default=50)
    ap.add_argument("--next-iters", type=int, default=50,
                    help="launches of each of cape_expand and glide_kv_compact timed after the step")
    ap.add_argument("--cpu-pairs", type=int, default=0,
                    help="(b, h) slabs in the CPU-baseline sample; 0 = every slab of one step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--config-steps", type=int, default=30,
                    help="timed rounds of each evaluation workload and of the CaPE rounds")
    ap.add_argument("--no-per-config", action="store_true",
                    help="skip the per-workload rounds and the CaPE rounds")
    ap.add_argument("--force-fma", action="store_true")
    ap.add_argument("--batch", type=int, default=0,
                    help="keep only the first N sequences of the workload (smaller profiling captures)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        return run_reference(args, rank, world)
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    return run_glide(args, rank, world, local_rank)


if __name__ == "__main__":
    sys.exit(main())
