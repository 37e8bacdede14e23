"""Element-by-element comparison of a whole translation against the oracle, split over
spawned processes by (target layer, sequence).

Each job carries one target layer's source caches (the mapped source layers, one sequence),
its translator matrices and the CUDA path's output for that layer and sequence; the worker
builds a one-layer, one-sequence oracle problem, translates it in fp64 and returns the
comparison's sums, so a full-size workload is checked on every output element in seconds.
The pool is started with `spawn` (safe after CUDA initialisation in the parent) and never
imports torch.
"""
from __future__ import annotations

import atexit
import dataclasses
import multiprocessing as mp
import os
from typing import Dict, List, Optional

import numpy as np

ABS_TOL = 3e-2
BF16_HALF_ULP_REL = 2.0 ** -8
REL_L2 = 1e-2

_pool = None


def pool():
    global _pool
    if _pool is None:
        n = max(1, min(16, (os.cpu_count() or 1)))
        _pool = mp.get_context("spawn").Pool(n)
        atexit.register(_pool.terminate)
    return _pool


def _bits(x: np.ndarray) -> np.ndarray:
    """Raw bf16 bits of float32 values that are exactly bf16 (lossless)."""
    from paper_2608_30963_gb300 import synth
    return synth.f32_to_bf16_bits(np.ascontiguousarray(x, np.float32))


def _unbits(b: np.ndarray) -> np.ndarray:
    from paper_2608_30963_gb300 import synth
    return synth.bf16_bits_to_f32(b)


@dataclasses.dataclass
class Job:
    src_geom: object          # ModelGeom (num_layers = number of mapped layers in src_k)
    dst_geom: object          # ModelGeom with num_layers = 1
    dtype: str
    form: int
    k_layers: int
    layer_row: List[int]      # source layers of this target layer, as indices into src_k / src_v
    src_k: List[np.ndarray]   # [1, Hs, S, ds] bf16 bits (uint16) or float32
    src_v: List[np.ndarray]
    src_len: int
    tgt_len: int
    span_lo: Optional[np.ndarray]
    span_hi: Optional[np.ndarray]
    src_pos: Optional[np.ndarray]
    tgt_pos: Optional[np.ndarray]
    w_k: Optional[np.ndarray]    # [1, Ht, in, dt] float32
    w_v: Optional[np.ndarray]
    low_rank: Optional[tuple]
    gpu_k: np.ndarray             # [Ht, T, dt] bf16 bits or float32
    gpu_v: np.ndarray
    tag: str = ""


def _f32(x):
    return _unbits(x) if x.dtype == np.uint16 else np.asarray(x, np.float32)


def _worker(job: Job) -> Dict:
    import oracle
    ks = [_f32(a) for a in job.src_k]
    vs = [_f32(a) for a in job.src_v]
    so = np.array([0, job.tgt_len], np.int32)
    p = oracle.OracleProblem(job.src_geom, job.dst_geom, np.asarray(job.layer_row, np.int32).reshape(1, -1),
                             np.array([job.src_len], np.int32), so, ks[0].shape[2], job.tgt_len, ks, vs,
                             job.w_k, job.w_v, job.span_lo, job.span_hi, job.src_pos, job.tgt_pos,
                             form=job.form, k_layers=job.k_layers, low_rank=job.low_rank)
    ok, ov = p.translate()                                       # [1, Ht, T, dt] float64
    out = {"tag": job.tag, "n": 0, "err_sq": 0.0, "ref_sq": 0.0, "max_abs": 0.0, "n_above_3e-2": 0,
           "n_bad": 0, "worst_excess": -np.inf, "finite": True}
    extra = [0.0, 0.0]
    if job.low_rank is not None:
        extra = [latent_fold_bound(p, job.low_rank, kv, job.tgt_len) for kv in (0, 1)]
    for (gpu, ref), ex in zip(((_f32(job.gpu_k), ok[0]), (_f32(job.gpu_v), ov[0])), extra):
        g = np.asarray(gpu, np.float64)
        if not np.all(np.isfinite(g)):
            out["finite"] = False
        err = np.abs(g - ref)
        out["n"] += int(err.size)
        out["err_sq"] += float((err * err).sum())
        out["ref_sq"] += float((ref * ref).sum())
        out["max_abs"] = max(out["max_abs"], float(err.max(initial=0.0)))
        out["n_above_3e-2"] += int((err > ABS_TOL).sum())
        bound = ABS_TOL + BF16_HALF_ULP_REL * np.abs(ref) if job.dtype == "bf16" else np.full_like(ref, ABS_TOL)
        bound = bound + ex
        ex = err - bound
        out["n_bad"] += int((ex > 0).sum())
        out["worst_excess"] = max(out["worst_excess"], float(ex.max(initial=-np.inf)))
    return out


def latent_fold_bound(p, low_rank, kv: int, T: int) -> np.ndarray:
    """A latent adapter x -> (x A) B is applied by the library as x W with W = A B folded at
    creation and rounded to bf16 (|W' - W| <= 2^-8 |W| elementwise), so its outputs may differ
    from the chained maps by up to 2^-8 sum_i |xbar_i| |W_io| beyond the bf16 tolerance; this is
    that bound per output element, [Ht, T, dt], from the oracle's input rows xbar."""
    a, b = low_rank[2 * kv], low_rank[2 * kv + 1]             # [1, Ht, in, rank], [1, Ht, rank, dt]
    Ht = a.shape[1]
    out = []
    for h in range(Ht):
        W = np.asarray(a[0, h], np.float64) @ np.asarray(b[0, h], np.float64)
        X = np.stack([p.input_row(0, h, kv, tp) for tp in range(T)])
        out.append(BF16_HALF_ULP_REL * (np.abs(X) @ np.abs(W)))
    return np.stack(out)


def run(jobs: List[Job]) -> Dict:
    """Runs the jobs and merges their sums into one comparison record (rel-L2 over all outputs,
    literal max-abs, elements above 3e-2, elements outside the element-wise bound)."""
    res = pool().map(_worker, jobs, chunksize=1)
    tot = {"n": 0, "err_sq": 0.0, "ref_sq": 0.0, "max_abs": 0.0, "n_above_3e-2": 0, "n_bad": 0,
           "worst_excess": -np.inf, "finite": True, "jobs": len(res)}
    for r in res:
        for k in ("n", "err_sq", "ref_sq", "n_above_3e-2", "n_bad"):
            tot[k] += r[k]
        tot["max_abs"] = max(tot["max_abs"], r["max_abs"])
        tot["worst_excess"] = max(tot["worst_excess"], r["worst_excess"])
        tot["finite"] = tot["finite"] and r["finite"]
    tot["rel_l2"] = float(np.sqrt(tot["err_sq"] / tot["ref_sq"])) if tot["ref_sq"] > 0 else float(np.sqrt(tot["err_sq"]))
    return tot


def check(tot: Dict, label: str = "") -> Dict:
    """Asserts the comparison record meets the tolerances and logs it."""
    from harness import record
    stats = {"rel_l2": tot["rel_l2"], "max_abs": tot["max_abs"], "n": tot["n"], "n_above_3e-2": tot["n_above_3e-2"]}
    record(stats, label)
    assert tot["finite"], "non-finite output"
    assert tot["rel_l2"] <= REL_L2, tot
    assert tot["n_bad"] == 0, tot
    return stats


def jobs_for(spec, wl, layer_map, src_k: Dict[int, np.ndarray], src_v: Dict[int, np.ndarray], w_k, w_v,
             gpu_layer, layers=None, low_rank=None, src_pos=None, tgt_pos=None) -> List[Job]:
    """One job per (target layer, sequence).

    src_k / src_v: source layer -> [B, Hs, S_max, ds] float32 (bf16-exact values for bf16).
    gpu_layer(j, kv) -> the CUDA path's target layer j as [Ht, T_total, dt] float32.
    layers: the target layers to check (default: all).
    """
    s, d = spec.src, spec.dst
    lm = np.asarray(layer_map, np.int32).reshape(d.num_layers, -1)
    kl = lm.shape[1]
    layers = range(d.num_layers) if layers is None else layers
    bf = spec.dtype == "bf16"
    enc = _bits if bf else (lambda x: np.ascontiguousarray(x, np.float32))
    jobs = []
    for j in layers:
        gk_all, gv_all = gpu_layer(j, 0), gpu_layer(j, 1)
        row = [int(x) for x in lm[j]]
        uniq = sorted(set(row))
        for b in range(wl.batch):
            S, a, e = int(wl.src_len[b]), int(wl.tgt_seq_off[b]), int(wl.tgt_seq_off[b + 1])
            if e == a:
                continue
            Sm = max(S, 1)
            ks = [enc(src_k[l][b:b + 1, :, :Sm]) for l in uniq]
            vs = [enc(src_v[l][b:b + 1, :, :Sm]) for l in uniq]
            lr = None
            if low_rank is not None:
                lr = tuple(np.ascontiguousarray(x[j:j + 1]) for x in low_rank)
            jobs.append(Job(
                src_geom=dataclasses.replace(s, num_layers=len(uniq)),
                dst_geom=dataclasses.replace(d, num_layers=1), dtype=spec.dtype, form=spec.form, k_layers=kl,
                layer_row=[uniq.index(x) for x in row], src_k=ks, src_v=vs, src_len=S, tgt_len=e - a,
                span_lo=None if wl.span_lo is None else np.ascontiguousarray(wl.span_lo[a:e]),
                span_hi=None if wl.span_hi is None else np.ascontiguousarray(wl.span_hi[a:e]),
                src_pos=None if src_pos is None else np.ascontiguousarray(np.asarray(src_pos)[b, :Sm]),
                tgt_pos=None if tgt_pos is None else np.ascontiguousarray(np.asarray(tgt_pos)[a:e]),
                w_k=None if w_k is None else np.ascontiguousarray(w_k[j:j + 1]),
                w_v=None if w_v is None else np.ascontiguousarray(w_v[j:j + 1]),
                low_rank=lr, gpu_k=enc(gk_all[:, a:e]), gpu_v=enc(gv_all[:, a:e]), tag=f"layer {j} seq {b}"))
    return jobs
