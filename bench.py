"""Benchmark: translated KV tokens/s and ms per handoff for cross-model KV translation.

One step = one kvx_translate call over the whole workload (all target layers,
heads, K and V, every target token): layer alignment, span gather, undo the
source RoPE, span mean, GQA-regrouped projection, target RoPE and target cache
write.  Default workload: Qwen2.5-7B-shaped -> Qwen2.5-1.5B-shaped KV caches,
4096 tokens, batch 1, bf16 (the within-family handoff of the paper's
Section 6.2 at the 4K context the headline metric names).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl kvx|reference] [--workload NAME]

Prints ONE JSON line on rank 0.  Under torchrun (N > 1) every rank translates
its own replica of the workload (no collective on the data path: the handoffs
are independent); the timed region is bracketed by barriers and the time is
the max over ranks.
"""
from __future__ import annotations

import argparse
import json
import math
import multiprocessing as mp
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_30963_gb300 import synth  # noqa: E402  (numpy only)

DEFAULT_WORKLOAD = "qwen7b_to_qwen1p5b_4k"
NOMINAL_HBM_GBS = 8000.0   # nominal HBM3e bandwidth of a GB300 (vendor figure, about 8 TB/s)
METRIC = "translated KV tokens/s and ms/handoff at 4K (7B→1.5B shapes); % of roofline"


# ----------------------------------------------------------------------------- workload arithmetic
def algorithmic(spec: synth.WorkloadSpec, wl: synth.Workload, layer_map) -> dict:
    """Bytes a translate must move at least once, and its FLOPs."""
    elt = 2 if spec.dtype == "bf16" else 4
    S_tot = int(wl.src_len.sum())
    T = wl.total_tgt
    src_layers = len(set(int(x) for x in np.asarray(layer_map).reshape(-1)))
    rd = src_layers * spec.src.num_kv_heads * S_tot * spec.src.head_dim * 2 * elt
    wr = spec.dst.num_layers * spec.dst.num_kv_heads * T * spec.dst.head_dim * 2 * elt
    # translator parameters: the full matrices, or a latent adapter's two factors
    per = spec.group_in * spec.dst.head_dim if spec.rank == 0 else spec.rank * (spec.group_in + spec.dst.head_dim)
    wt = 2 * spec.dst.num_layers * spec.dst.num_kv_heads * per * elt
    flops = 2.0 * T * spec.group_in * spec.dst.head_dim * spec.dst.num_layers * spec.dst.num_kv_heads * 2
    return {"read": rd, "write": wr, "weights": wt, "bytes": rd + wr + wt, "flops": flops}


def aggregate(elapsed_ms: float, tokens_per_step: int, steps: int, world: int, dist=None, device=None):
    """Whole-job throughput: every rank translates its own replica; the job time
    is the slowest rank's.  Returns (max elapsed ms, tokens/s over all ranks)."""
    if dist is not None and world > 1:
        import torch
        t = torch.tensor([float(elapsed_ms)], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        elapsed_ms = float(t.item())
    return elapsed_ms, tokens_per_step * steps * world / (elapsed_ms / 1e3)


def nearest_map(Ls, Lt):
    return [0] * Lt if Lt == 1 else [(2 * j * (Ls - 1) + (Lt - 1)) // (2 * (Lt - 1)) for j in range(Lt)]


# ----------------------------------------------------------------------------- CPU oracle (baseline / reference arm)
def _oracle_worker(args):
    """Time the oracle on target rows [t0, t0+n) of layer 0, K and V, all heads.

    Runs in a spawned process; imports the oracle there."""
    name, t0, n, budget_s = args
    import oracle
    spec = synth.config_specs()[name]
    wl = synth.make_workload(spec)
    lm = wl.layer_map if wl.layer_map is not None else oracle.layer_map_nearest(spec.src.num_layers,
                                                                                spec.dst.num_layers)
    l0 = int(np.asarray(lm).reshape(-1)[0])
    k = synth.source_kv(wl, l0, 0)
    if spec.src.rope_base > 0:
        k = oracle.rope_cache(k, spec.src)
        if spec.dtype == "bf16":
            k = synth.bf16_round(k)
    v = synth.source_kv(wl, l0, 1)
    ks = [k] * spec.src.num_layers
    vs = [v] * spec.src.num_layers
    if spec.rank > 0:
        low_rank, wk, wv = (*synth.latent_factors(wl, 0), *synth.latent_factors(wl, 1)), None, None
    else:
        low_rank, wk, wv = None, synth.weights(wl, 0), synth.weights(wl, 1)
    p = oracle.OracleProblem(spec.src, spec.dst, lm, wl.src_len, wl.tgt_seq_off, wl.s_max, wl.t_max, ks, vs,
                             wk, wv, wl.span_lo, wl.span_hi, form=spec.form, k_layers=spec.layers_per_target,
                             low_rank=low_rank)
    rows = 0
    start = time.perf_counter()
    T = wl.total_tgt
    i = 0
    while True:
        tp = (t0 + i) % T
        for h in range(spec.dst.num_kv_heads):
            for kv in (0, 1):
                p.row(0, h, kv, tp)
                rows += 1
        i += 1
        el = time.perf_counter() - start
        if (n and i >= n) or (not n and el >= budget_s):
            break
    return rows, time.perf_counter() - start


def cpu_baseline(pool, name: str, budget_s: float, cores: int) -> dict:
    """Oracle throughput on the host cores, as target tokens/s (one target token
    = L_t * H_t * 2 output rows)."""
    spec = synth.config_specs()[name]
    args = [(name, 97 * i, 0, budget_s) for i in range(cores)]
    t0 = time.perf_counter()
    res = pool.map(_oracle_worker, args)
    wall = time.perf_counter() - t0
    rows = sum(r for r, _ in res)
    busy = max(t for _, t in res)
    rows_per_tok = spec.dst.num_layers * spec.dst.num_kv_heads * 2
    tok_s = rows / busy / rows_per_tok
    return {"value": tok_s, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"{rows} output rows (target layer 0, all heads, K and V) of workload {name}, "
                      f"{budget_s:.0f} s per core on {cores} spawned processes; scaled to tokens by "
                      f"{rows_per_tok} rows per target token",
            "wall_s": wall}


# ----------------------------------------------------------------------------- clocks
CLOCK_Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
           "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
           "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


class ClockSampler:
    def __init__(self, gpu_index: int):
        self.proc = None
        self.path = None
        try:
            self.path = os.path.join(tempfile.gettempdir(), f"kvx_clocks_{os.getpid()}.csv")
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={CLOCK_Q}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for nm, val in zip(names, parts[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(nm)
        try:
            os.remove(self.path)
        except OSError:
            pass
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ----------------------------------------------------------------------------- input synthesis
def rotate_np(x: np.ndarray, base: float) -> np.ndarray:
    """Apply half-split RoPE (plain frequency schedule) at positions 0..S-1 (input
    synthesis: the post-RoPE keys a source model's prefill stores)."""
    B, H, S, d = x.shape
    h = d // 2
    ang = np.arange(S, dtype=np.float64)[:, None] * np.power(base, -2.0 * np.arange(h) / d)[None, :]
    c, s = np.cos(ang), np.sin(ang)
    x0, x1 = x[..., :h].astype(np.float64), x[..., h:].astype(np.float64)
    return np.concatenate([x0 * c - x1 * s, x1 * c + x0 * s], axis=-1).astype(np.float32)


def to_torch(x: np.ndarray, dtype: str, torch, pin=False):
    if dtype == "bf16":
        t = torch.from_numpy(synth.f32_to_bf16_bits(x).view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(x, np.float32))
    return t.pin_memory() if pin else t


# ----------------------------------------------------------------------------- main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="kvx", choices=["kvx", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--cpu-budget", type=float, default=12.0, help="seconds of oracle work per core")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--mode", default="translate", choices=["translate", "fit"],
                    help="translate: the hot path (default); fit: the closed-form translator fit's accumulation")
    ap.add_argument("--record-traffic", metavar="CSV",
                    help="maintenance (no GPU): write profiles/traffic.json from an ncu --csv capture of one "
                         "identity-kernel launch of --workload")
    ap.add_argument("--traffic-command", default="", help="the ncu command that produced --record-traffic's CSV")
    ap.add_argument("--traffic-rev", default="", help="git revision whose sources the captured kernel was built from")
    args = ap.parse_args()
    if args.record_traffic:
        return record_traffic(args.record_traffic, args.workload, args.traffic_command, args.traffic_rev)
    args.warmup = max(args.warmup, 3)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    spec = synth.config_specs()[args.workload]

    if args.impl == "reference":
        return reference_arm(args, spec, rank, world)
    if args.mode == "fit":
        return fit_bench(args, spec)

    # spawn the oracle pool before any CUDA call
    pool = None
    cores = os.cpu_count() or 1
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        pool = mp.get_context("spawn").Pool(cores)

    import torch
    import paper_2608_30963_gb300 as kvx

    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))

    wl = synth.make_workload(spec)
    lm = wl.layer_map.tolist() if wl.layer_map is not None else nearest_map(spec.src.num_layers, spec.dst.num_layers)
    alg = algorithmic(spec, wl, lm)
    tdt = torch.bfloat16 if spec.dtype == "bf16" else torch.float32
    kdt = kvx.KVX_BF16 if spec.dtype == "bf16" else kvx.KVX_FP32

    # host inputs (pinned) and the translator
    mapped = sorted(set(int(x) for x in np.asarray(lm).reshape(-1)))
    host_k, host_v = {}, {}
    for l in mapped:
        k = synth.source_kv(wl, l, 0)
        if spec.src.rope_base > 0:
            if spec.src.rope_type != synth.ROPE_DEFAULT:
                raise SystemExit("bench input synthesis rotates with the plain RoPE schedule only")
            k = rotate_np(k, spec.src.rope_base)
        host_k[l] = to_torch(k, spec.dtype, torch, pin=True)
        host_v[l] = to_torch(synth.source_kv(wl, l, 1), spec.dtype, torch, pin=True)
    if spec.rank > 0:
        (a_k, b_k), (a_v, b_v) = synth.latent_factors(wl, 0), synth.latent_factors(wl, 1)
        tr = kvx.Translator(spec.src, spec.dst, None, None, layer_map=lm, dtype=kdt, form=spec.form,
                            layers_per_target=spec.layers_per_target,
                            low_rank=tuple(to_torch(x, spec.dtype, torch) for x in (a_k, b_k, a_v, b_v)))
    else:
        tr = kvx.Translator(spec.src, spec.dst, to_torch(synth.weights(wl, 0), spec.dtype, torch),
                            to_torch(synth.weights(wl, 1), spec.dtype, torch), layer_map=lm, dtype=kdt,
                            form=spec.form, layers_per_target=spec.layers_per_target)
    info = tr.info()

    dev = torch.device("cuda", local_rank)
    i32 = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(dev)
    src_len, seq_off = i32(wl.src_len), i32(wl.tgt_seq_off)
    span_lo, span_hi = i32(wl.span_lo), i32(wl.span_hi)
    page_table = i32(wl.page_table) if spec.paged else None
    # cross-tokenizer workloads: every step first builds the token-span alignment on the device
    # from the two tokenisations' byte offsets (kvx_build_alignment), then translates with it
    align = None
    if spec.cross_tokenizer:
        align = dict(src_seq_off=i32(wl.src_seq_off), src_end=i32(wl.src_end), tgt_seq_off=seq_off,
                     tgt_end=i32(wl.tgt_end), span_lo=torch.empty_like(span_lo), span_hi=torch.empty_like(span_hi))
        span_lo, span_hi = align["span_lo"], align["span_hi"]
        # the builder reads both byte-offset arrays and the sequence offsets, writes two span arrays
        alg["bytes"] += 4 * (int(wl.src_end.size) + 3 * int(wl.tgt_end.size) + 2 * (wl.batch + 1))
    Lt, Ht, dt = spec.dst.num_layers, spec.dst.num_kv_heads, spec.dst.head_dim
    out_shape = (wl.num_pages, spec.page_size, Ht, dt) if spec.paged else (wl.batch, Ht, wl.t_max, dt)

    # rotating input/output sets so that consecutive steps share nothing in L2
    l2_bytes = 129 * 2 ** 20
    set_bytes = alg["read"] + alg["write"]
    nsets = max(2, min(8, math.ceil(4 * l2_bytes / set_bytes)))
    sets = []
    for _ in range(nsets):
        sk = {l: host_k[l].to(dev) for l in mapped}
        sv = {l: host_v[l].to(dev) for l in mapped}
        src_k = [sk.get(l, sk[mapped[0]]) for l in range(spec.src.num_layers)]
        src_v = [sv.get(l, sv[mapped[0]]) for l in range(spec.src.num_layers)]
        dk = [torch.empty(out_shape, dtype=tdt, device=dev) for _ in range(Lt)]
        dv = [torch.empty(out_shape, dtype=tdt, device=dev) for _ in range(Lt)]
        sets.append((src_k, src_v, dk, dv))
    stream = torch.cuda.current_stream()

    def build_spans(stream_=None):
        if align is not None:
            kvx.build_alignment(align["src_seq_off"], align["src_end"], align["tgt_seq_off"], align["tgt_end"],
                                align["span_lo"], align["span_hi"], stream=stream_)

    def step(i):
        src_k, src_v, dk, dv = sets[i % nsets]
        build_spans()
        tr.translate(src_k, src_v, src_len, seq_off, wl.total_tgt, dk, dv, span_lo=span_lo, span_hi=span_hi,
                     page_table=page_table, page_size=spec.page_size, num_pages=wl.num_pages, stream=None)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    if tr.device_status() != 0:
        raise RuntimeError("device status nonzero after warm-up")
    # kvx_translate allocates nothing and never synchronises, so the K timed steps
    # (input sets alternating) are captured as one CUDA graph: the host leaves the
    # timed loop, and consecutive translates overlap launch and on-chip set-up
    # (programmatic dependent launch) while keeping stream order for memory.
    def capture(n):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for i in range(n):
                step(i)
        return g

    g_warm = capture(args.warmup)
    g_timed = capture(args.steps)
    g_warm.replay()
    torch.cuda.synchronize()

    clocks = ClockSampler(local_rank)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    g_timed.replay()
    t_end.record(stream)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    elapsed_ms = t_start.elapsed_time(t_end)
    launch_ms = [elapsed_ms / args.steps]   # one step's launches, back to back

    # keep the GPU loaded long enough for the clock sampler to see it (>= 1 s)
    extra = 0
    t0 = time.perf_counter()
    while time.perf_counter() - t0 < 1.0:
        g_timed.replay()
        torch.cuda.synchronize()
        extra += args.steps
    clk = clocks.stop()
    if tr.device_status() != 0:
        raise RuntimeError("device status nonzero after the timed region")

    elapsed_ms, value = aggregate(elapsed_ms, wl.total_tgt, args.steps, world, dist, dev)

    # end to end through the C ABI with host buffers: every step copies its source caches in from
    # pinned host memory, translates, and copies the target caches out.  Consecutive steps overlap
    # on three streams (copy in, translate, copy out) over two device buffer sets and two host
    # output sets, as a serving loop streaming handoffs would.
    e2e_steps = max(1, args.e2e_steps)
    host_out = [[torch.empty(out_shape, dtype=tdt).pin_memory() for _ in range(2 * Lt)] for _ in range(2)]
    h2d = sum(host_k[l].numel() * host_k[l].element_size() * 2 for l in mapped)
    host_ends = None
    if align is not None:   # the two tokenisations' byte offsets are inputs of every step too
        host_ends = (torch.from_numpy(np.ascontiguousarray(wl.src_end, np.int32)).pin_memory(),
                     torch.from_numpy(np.ascontiguousarray(wl.tgt_end, np.int32)).pin_memory())
        h2d += 4 * (int(wl.src_end.size) + int(wl.tgt_end.size))
    d2h = sum(t.numel() * t.element_size() for t in sets[0][2]) * 2
    s_in, s_tr, s_out = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    ev = lambda: torch.cuda.Event()
    in_done, tr_done, out_done = [ev(), ev()], [ev(), ev()], [ev(), ev()]
    used = [False, False]

    def e2e_step(i):
        k = i % 2
        src_k, src_v, dk, dv = sets[k]
        if used[k]:
            s_in.wait_event(tr_done[k])       # the translate of step i-2 has read this source set
            s_tr.wait_event(out_done[k])      # the copy-out of step i-2 has read this target set
        with torch.cuda.stream(s_in):
            for l in mapped:
                src_k[l].copy_(host_k[l], non_blocking=True)
                src_v[l].copy_(host_v[l], non_blocking=True)
            if host_ends is not None:   # one device copy of the offsets: every step writes the same values
                align["src_end"].copy_(host_ends[0], non_blocking=True)
                align["tgt_end"].copy_(host_ends[1], non_blocking=True)
            in_done[k].record(s_in)
        s_tr.wait_event(in_done[k])
        build_spans(s_tr)
        tr.translate(src_k, src_v, src_len, seq_off, wl.total_tgt, dk, dv, span_lo=span_lo, span_hi=span_hi,
                     page_table=page_table, page_size=spec.page_size, num_pages=wl.num_pages, stream=s_tr)
        tr_done[k].record(s_tr)
        s_out.wait_event(tr_done[k])
        with torch.cuda.stream(s_out):
            for j in range(Lt):
                host_out[k][j].copy_(dk[j], non_blocking=True)
                host_out[k][Lt + j].copy_(dv[j], non_blocking=True)
            out_done[k].record(s_out)
        used[k] = True

    for s_ in (s_in, s_tr, s_out):
        s_.wait_stream(stream)
    e2e_step(0)
    e2e_step(1)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(s_in)
    for i in range(e2e_steps):
        e2e_step(i)
    s_in.wait_stream(s_out)
    b.record(s_in)
    torch.cuda.synchronize()
    e2e_ms = a.elapsed_time(b)
    e2e_ms, e2e_value = aggregate(e2e_ms, wl.total_tgt, e2e_steps, world, dist, dev)
    if tr.device_status() != 0:
        raise RuntimeError("device status nonzero after the end-to-end steps")

    # the host-link ceiling of the same copies with no translation: H2D alone, D2H alone, and
    # both directions at once on two streams (what the overlapped end-to-end steps need per step)
    def timed_copies(h2d_on, d2h_on, reps=3):
        best = float("inf")
        src_k, src_v, dk, dv = sets[0]
        for _ in range(reps):
            torch.cuda.synchronize()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(s_in)
            s_out.wait_stream(s_in)
            if h2d_on:
                with torch.cuda.stream(s_in):
                    for l in mapped:
                        src_k[l].copy_(host_k[l], non_blocking=True)
                        src_v[l].copy_(host_v[l], non_blocking=True)
            if d2h_on:
                with torch.cuda.stream(s_out):
                    for j in range(Lt):
                        host_out[0][j].copy_(dk[j], non_blocking=True)
                        host_out[0][Lt + j].copy_(dv[j], non_blocking=True)
            s_in.wait_stream(s_out)
            b.record(s_in)
            torch.cuda.synchronize()
            best = min(best, a.elapsed_time(b))
        return best

    h2d_ms, d2h_ms, both_ms = timed_copies(True, False), timed_copies(False, True), timed_copies(True, True)
    copy_ceiling = {"h2d_ms": h2d_ms, "d2h_ms": d2h_ms, "both_ms": both_ms,
                    "h2d_gbs": h2d / (h2d_ms / 1e3) / 1e9, "d2h_gbs": d2h / (d2h_ms / 1e3) / 1e9,
                    "tokens_per_s": wl.total_tgt / (both_ms / 1e3),
                    "how": "the step's pinned copies alone (no translation), best of 3: H2D, D2H, and both "
                           "directions at once on two streams; tokens_per_s = target tokens / both_ms"}

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return

    T = wl.total_tgt
    ms_step = elapsed_ms / args.steps
    avg_launch_ms = statistics.mean(launch_ms)
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        pass
    hbm_peak = peaks.get("hbm_gbs")
    peak_src = "measured" if hbm_peak else "fallback"
    hbm_peak = hbm_peak or 6800.0
    achieved = alg["bytes"] / (avg_launch_ms / 1e3) / 1e9
    traffic = traffic_for(args.workload)
    line = {
        "metric": METRIC,
        "value": value,
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms_step,
        "ms_per_handoff": ms_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": spec.dtype,
        "data": "synthetic",
        "config": {"workload": args.workload,
                   "src": f"L{spec.src.num_layers} H{spec.src.num_kv_heads} d{spec.src.head_dim} base{spec.src.rope_base:g}",
                   "dst": f"L{spec.dst.num_layers} H{spec.dst.num_kv_heads} d{spec.dst.head_dim} base{spec.dst.rope_base:g}",
                   "target_tokens": T, "batch": wl.batch, "paged": spec.paged,
                   "l2": f"inputs larger than L2: {nsets} rotating input/output sets of {set_bytes / 1e6:.1f} MB "
                         f"(L2 129 MB)",
                   "parallelism": f"replicas{world}" if world > 1 else "single",
                   "step": ("kvx_build_alignment (byte offsets -> spans) + kvx_translate" if align is not None
                            else "kvx_translate (same tokenizer: identity alignment)"),
                   "timing": "the K steps as one CUDA graph (programmatic dependent launch between steps); "
                             "CUDA events around it"},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                     "frac": achieved / hbm_peak, "traffic": traffic,
                     "peak_source": f"{peak_src} hbm_gbs (copy)",
                     # the same achieved bandwidth against the nominal HBM3e figure (about 8 TB/s)
                     "nominal_peak": NOMINAL_HBM_GBS, "frac_nominal": achieved / NOMINAL_HBM_GBS,
                     "algorithmic_bytes_per_launch": alg["bytes"], "avg_launch_ms": avg_launch_ms,
                     "tensor_tflops": alg["flops"] / (avg_launch_ms / 1e3) / 1e12},
        "clocks": clk,
        "e2e": {"value": e2e_value, "unit": "tokens/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms / e2e_steps,
                "how": ("per step: H2D of the source caches " +
                        ("and both tokenisations' byte offsets " if align is not None else "") +
                        "from pinned memory, " +
                        ("kvx_build_alignment, " if align is not None else "") +
                        "kvx_translate, D2H of the target caches; consecutive steps overlap on three streams "
                        "over two buffer sets"),
                "copy_ceiling": copy_ceiling,
                "frac_of_copy_ceiling": e2e_value / copy_ceiling["tokens_per_s"]},
        "gpu_launches": args.steps * (tr.launches_per_translate() + (1 if align is not None else 0)),
        "kernel_path": ({1: "simt", 2: "tcgen05"}.get(info.path, str(info.path)) +
                        ("+tma_identity" if info.path == 2 and span_lo is None else "")),
        "num_sms": info.num_sms,
    }
    if pool is not None:
        line["cpu_baseline"] = cpu_baseline(pool, args.workload, args.cpu_budget, cores)
        pool.close()
    print(json.dumps(line), flush=True)
    tr.close()
    if dist:
        dist.destroy_process_group()


def _oracle_fit_worker(args):
    """Time the oracle's fit on a sub-problem: target layer 0, head 0 (K and V), the workload's
    first n_tok target tokens.  Runs in a spawned process."""
    name, n_tok = args
    import dataclasses as dc
    import oracle
    spec = synth.config_specs()[name]
    wl = synth.make_workload(spec, [n_tok])
    lm = wl.layer_map if wl.layer_map is not None else oracle.layer_map_nearest(spec.src.num_layers,
                                                                                spec.dst.num_layers)
    lm = np.asarray(lm).reshape(spec.dst.num_layers, -1)[:1]
    k = synth.source_kv(wl, int(lm.reshape(-1)[0]), 0)
    v = synth.source_kv(wl, int(lm.reshape(-1)[0]), 1)
    dst = dc.replace(spec.dst, num_layers=1, num_kv_heads=1)
    src = spec.src if spec.src.num_kv_heads >= spec.dst.num_kv_heads else dc.replace(spec.src, num_kv_heads=1)
    src = dc.replace(src, num_kv_heads=min(src.num_kv_heads, spec.heads_per_layer if spec.form else
                                           max(1, spec.src.num_kv_heads // spec.dst.num_kv_heads)))
    k, v = k[:, :src.num_kv_heads], v[:, :src.num_kv_heads]
    ks, vs = [k] * spec.src.num_layers, [v] * spec.src.num_layers
    rng = np.random.default_rng(0)
    tk = [rng.standard_normal((1, 1, wl.t_max, dst.head_dim)).astype(np.float32)]
    tv = [rng.standard_normal((1, 1, wl.t_max, dst.head_dim)).astype(np.float32)]
    z = np.zeros((1, 1, spec.group_in, dst.head_dim), np.float32)
    p = oracle.OracleProblem(src, dst, lm, wl.src_len, wl.tgt_seq_off, wl.s_max, wl.t_max, ks, vs, z, z,
                             wl.span_lo, wl.span_hi, form=spec.form, k_layers=spec.layers_per_target)
    t0 = time.perf_counter()
    p.fit(tk, tv, 1e-3)
    return time.perf_counter() - t0


def fit_bench(args, spec):
    """Closed-form fit: calibration tokens/s of kvx_fit_accumulate (input rows, target rows, Gram
    sums) over the workload, plus one solve.  Inputs resident on the device."""
    # the oracle's fit timed on the host cores (spawned before any CUDA call): one (layer, head)
    # pair of systems per process over up to 4096 tokens, scaled to all groups
    cores = os.cpu_count() or 1
    n_tok = min(4096, int(sum(spec.tgt_lens)))
    total_groups = spec.dst.num_layers * spec.dst.num_kv_heads
    cpu_tok_s = None
    if not args.no_cpu_baseline:
        with mp.get_context("spawn").Pool(cores) as pool:
            secs = pool.map(_oracle_fit_worker, [(args.workload, n_tok)] * cores)
        groups_per_proc = 1   # one target layer, one head: a K and a V system
        cpu_tok_s = n_tok * cores * groups_per_proc / max(secs) / total_groups
    import torch
    import paper_2608_30963_gb300 as kvx
    torch.cuda.set_device(0)
    wl = synth.make_workload(spec)
    lm = wl.layer_map.tolist() if wl.layer_map is not None else nearest_map(spec.src.num_layers, spec.dst.num_layers)
    dev = torch.device("cuda", 0)
    g = torch.Generator(device=dev).manual_seed(0)
    s, d = spec.src, spec.dst
    mapped = sorted(set(int(x) for x in np.asarray(lm).reshape(-1)))
    shape = (wl.batch, s.num_kv_heads, wl.s_max, s.head_dim)
    ks = {l: torch.randn(shape, generator=g, device=dev).to(torch.bfloat16) for l in mapped}
    vs = {l: torch.randn(shape, generator=g, device=dev).to(torch.bfloat16) for l in mapped}
    src_k = [ks.get(l, ks[mapped[0]]) for l in range(s.num_layers)]
    src_v = [vs.get(l, vs[mapped[0]]) for l in range(s.num_layers)]
    tshape = (wl.batch, d.num_kv_heads, wl.t_max, d.head_dim)
    tk = [torch.randn(tshape, generator=g, device=dev).to(torch.bfloat16) for _ in range(d.num_layers)]
    tv = [torch.randn(tshape, generator=g, device=dev).to(torch.bfloat16) for _ in range(d.num_layers)]
    i32 = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(dev)
    src_len, seq_off = i32(wl.src_len), i32(wl.tgt_seq_off)
    span_lo, span_hi = i32(wl.span_lo), i32(wl.span_hi)
    f = kvx.Fitter(s, d, 1e-3, layer_map=lm, form=spec.form, layers_per_target=spec.layers_per_target)
    T = wl.total_tgt

    def step():
        f.accumulate(src_k, src_v, src_len, seq_off, T, tk, tv, span_lo=span_lo, span_hi=span_hi)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(args.steps):
        step()
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / args.steps
    wk = torch.empty((d.num_layers, d.num_kv_heads, spec.group_in, d.head_dim), dtype=torch.bfloat16, device=dev)
    wv = torch.empty_like(wk)
    t0 = time.perf_counter()
    bits = f.solve(wk, wv)
    solve_ms = (time.perf_counter() - t0) * 1e3
    elt = 2
    groups = d.num_layers * d.num_kv_heads * 2
    src_bytes = len(mapped) * s.num_kv_heads * int(wl.src_len.sum()) * s.head_dim * 2 * elt
    tgt_bytes = d.num_layers * d.num_kv_heads * T * d.head_dim * 2 * elt
    sums = groups * spec.group_in * (spec.group_in + d.head_dim) * 4 * 2
    flops = groups * T * 2.0 * spec.group_in * (spec.group_in + d.head_dim)
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        pass
    hbm, tc = peaks.get("hbm_gbs", 6800.0), peaks.get("bf16_tflops", 1900.0)
    byts = src_bytes + tgt_bytes + sums
    t_roof = max(byts / (hbm * 1e9), flops / (tc * 1e12))
    line = {"metric": "fit calibration tokens/s (kvx_fit_accumulate)", "value": T / (ms / 1e3), "unit": "tokens/s",
            "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "dtype": spec.dtype, "data": "synthetic", "mode": "fit",
            "config": {"workload": args.workload, "target_tokens": T, "groups": groups, "in": spec.group_in,
                       "lambda": 1e-3},
            "roofline": {"bound": "hbm" if byts / (hbm * 1e9) >= flops / (tc * 1e12) else "tensor",
                         "algorithmic_bytes": byts, "flops": flops, "roofline_ms": t_roof * 1e3,
                         "frac": t_roof * 1e3 / ms, "achieved_tflops": flops / (ms / 1e3) / 1e12,
                         "peaks": {"hbm_gbs": hbm, "bf16_tflops": tc}},
            "solve_ms": solve_ms, "solve_status": bits}
    if cpu_tok_s is not None:
        line["cpu_baseline"] = {"value": cpu_tok_s, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                                "sample": f"oracle fit (fp64 Gram sums and Cholesky) of target layer 0, head 0, K and "
                                          f"V over {n_tok} tokens in each of {cores} spawned processes, scaled by "
                                          f"{total_groups} (layer, head) pairs"}
    print(json.dumps(line), flush=True)
    f.close()


def kernel_rev(sources=None, rev: str = "") -> str:
    """Hash of the sources a kernel is compiled from (its translation unit and the headers it
    includes, paths relative to the repository root; all kernel sources when None), so a stored
    ncu traffic figure is only used for the kernel it measured."""
    import hashlib
    h = hashlib.sha1()
    if sources is None:
        csrc = os.path.join("paper_2608_30963_gb300", "csrc")
        sources = [os.path.join(csrc, f) for f in sorted(os.listdir(os.path.join(ROOT, csrc)))
                   if f.endswith((".cu", ".cuh", ".h"))]
    for f in sources:
        if rev:
            h.update(subprocess.check_output(["git", "-C", ROOT, "show", f"{rev}:{f}"]))
        else:
            h.update(open(os.path.join(ROOT, f), "rb").read())
    return h.hexdigest()[:12]


_TRAFFIC_REC = os.path.join(ROOT, "profiles", "traffic.json")
_TRAFFIC_SOURCES = ["paper_2608_30963_gb300/csrc/kvx_tc_aligned.cu", "paper_2608_30963_gb300/csrc/kvx_tc_common.cuh",
                    "paper_2608_30963_gb300/csrc/kvx_common.cuh", "paper_2608_30963_gb300/csrc/kvx_kernels.h",
                    "paper_2608_30963_gb300/csrc/kvx_schedule.h", "include/kvx.h"]
_UNITS = {"byte": 1, "kbyte": 1e3, "mbyte": 1e6, "gbyte": 1e9, "nsecond": 1e-9, "usecond": 1e-6,
          "msecond": 1e-3, "second": 1, "ns": 1e-9, "us": 1e-6, "ms": 1e-3, "s": 1}


def traffic_for(workload: str, rec_path: str = "") -> "int | None":
    """DRAM bytes of one identity-kernel launch from the traffic record, or None when the record
    is for another workload or the kernel's sources have changed since the capture."""
    try:
        rec = json.load(open(rec_path or _TRAFFIC_REC))
    except Exception:
        return None
    if rec.get("workload") != workload or rec.get("kernel_rev") != kernel_rev(rec.get("sources")):
        return None
    return rec.get("dram_bytes_per_launch")


def record_traffic(csv_path: str, workload: str, command: str, rev: str = "") -> int:
    """Writes profiles/traffic.json from the CSV that `ncu --csv --metrics
    gpu__time_duration.sum,dram__bytes_read.sum,dram__bytes_write.sum -k regex:aligned -c 1`
    printed for one launch of the identity-alignment kernel, keyed to the hash of the kernel's
    sources as they are now, or as git revision `rev` holds them when the capture ran on that
    revision (a later change to them leaves the bench's traffic null)."""
    import csv
    rows = [r for r in csv.reader(l for l in open(csv_path) if l.startswith('"'))]
    head, body = rows[0], rows[1:]
    col = {n: i for i, n in enumerate(head)}
    vals = {}
    kernel = None
    for r in body:
        if "aligned" not in r[col["Kernel Name"]]:
            continue
        if kernel is None:
            kernel = (r[col["ID"]], r[col["Kernel Name"]])
        if r[col["ID"]] != kernel[0]:
            continue
        v = float(r[col["Metric Value"]].replace(",", ""))
        vals[r[col["Metric Name"]]] = v * _UNITS.get(r[col["Metric Unit"]].lower(), 1)
    need = ("dram__bytes_read.sum", "dram__bytes_write.sum")
    if kernel is None or any(n not in vals for n in need):
        print("no identity-kernel launch with DRAM counters in", csv_path)
        return 1
    rec = {"workload": workload, "kernel": kernel[1].split("(")[0].split("::")[-1],
           "kernel_rev": kernel_rev(_TRAFFIC_SOURCES, rev),
           "dram_bytes_per_launch": int(round(vals[need[0]] + vals[need[1]])),
           "dram_bytes_read": int(round(vals[need[0]])), "dram_bytes_write": int(round(vals[need[1]])),
           "duration_s": vals.get("gpu__time_duration.sum"), "source": command,
           "note": "dram__bytes_read.sum + dram__bytes_write.sum of one launch (writes still resident in L2 "
                   "when the launch ends are not counted); kernel_rev hashes the listed sources",
           "sources": _TRAFFIC_SOURCES}
    with open(_TRAFFIC_REC, "w") as f:
        json.dump(rec, f, indent=1)
        f.write("\n")
    print(json.dumps(rec))
    return 0


def reference_arm(args, spec, rank, world):
    """The oracle as the reference implementation, timed on the host cores."""
    if rank != 0:
        return
    cores = os.cpu_count() or 1
    pool = mp.get_context("spawn").Pool(cores)
    budget = max(1.0, min(10.0, 120.0 / (args.steps + args.warmup)))
    for _ in range(args.warmup):
        pool.map(_oracle_worker, [(args.workload, 13 * i, 2, 0) for i in range(cores)])
    vals = []
    for _ in range(args.steps):
        cb = cpu_baseline(pool, args.workload, budget, cores)
        vals.append(cb["value"])
    pool.close()
    value = statistics.mean(vals)
    wl = synth.make_workload(spec)
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "impl": "reference", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": wl.total_tgt / value * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": args.workload, "target_tokens": wl.total_tgt},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": cb["sample"]},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
