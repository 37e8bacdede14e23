"""Shared test helpers: build one workload for both the CUDA path and the oracle.

The source K handed to both sides is the generator's pre-RoPE K rotated by the
oracle's RoPE (in double) and rounded to the storage type, i.e. the post-RoPE
cache a source model would hold.  Both sides then see bit-identical inputs.
"""
from __future__ import annotations

import dataclasses
import os
from typing import Dict, List, Optional, Sequence

import numpy as np

import oracle
from paper_2608_30963_gb300 import synth

# Tolerances for bf16 outputs: relative L2 <= 1e-2 over the whole output, and
# elementwise |gpu - ref| <= 3e-2 + 2^-8 |ref| (3e-2 plus the half-ulp of the
# bf16 store, which alone exceeds 3e-2 once |ref| >= 8).
REL_L2 = 1e-2
ABS_TOL = 3e-2
BF16_HALF_ULP_REL = 2.0 ** -8


@dataclasses.dataclass
class Case:
    wl: synth.Workload
    src_k: Dict[int, np.ndarray]       # source layer -> stored (post-RoPE) K, float32 values
    src_v: Dict[int, np.ndarray]
    w_k: np.ndarray
    w_v: np.ndarray
    layer_map: np.ndarray
    src_pos: Optional[np.ndarray] = None   # [B, S_max]
    tgt_pos: Optional[np.ndarray] = None   # [T_total]
    low_rank: Optional[tuple] = None       # (A_K, B_K, A_V, B_V) latent adapter factors

    @property
    def spec(self):
        return self.wl.spec


def make_case(spec: synth.WorkloadSpec, tgt_lens=None, layers: Optional[Sequence[int]] = None,
              pad_value: float = 0.0, src_pos=None, tgt_pos=None, wl: Optional[synth.Workload] = None) -> Case:
    """Inputs of one workload (wl: a prepared workload, e.g. with spans from two independent
    tokenisations; default: the spec's own)."""
    wl = synth.make_workload(spec, tgt_lens) if wl is None else wl
    lm = wl.layer_map if wl.layer_map is not None else oracle.layer_map_nearest(spec.src.num_layers,
                                                                                spec.dst.num_layers)
    need = sorted(set(int(x) for x in np.asarray(lm).reshape(-1))) if layers is None else sorted(set(layers))
    ks, vs = {}, {}
    for l in need:
        k = synth.source_kv(wl, l, 0, pad_value)
        if spec.src.rope_base > 0:
            pos = None if src_pos is None else np.asarray(src_pos, np.int32)
            k = oracle.rope_cache(k, spec.src, pos, +1)
        if spec.dtype == "bf16":
            k = synth.bf16_round(k)
        if pad_value != 0.0:
            for b in range(wl.batch):
                k[b, :, int(wl.src_len[b]):, :] = pad_value
        ks[l] = k
        vs[l] = synth.source_kv(wl, l, 1, pad_value)
    low_rank = None
    if spec.rank > 0:
        a_k, b_k = synth.latent_factors(wl, 0)
        a_v, b_v = synth.latent_factors(wl, 1)
        low_rank = (a_k, b_k, a_v, b_v)
        w_k = w_v = None
    else:
        w_k, w_v = synth.weights(wl, 0), synth.weights(wl, 1)
    return Case(wl, ks, vs, w_k, w_v, np.asarray(lm, np.int32),
                None if src_pos is None else np.asarray(src_pos, np.int32),
                None if tgt_pos is None else np.asarray(tgt_pos, np.int32), low_rank)


def oracle_problem(c: Case) -> oracle.OracleProblem:
    s = c.spec
    any_l = next(iter(c.src_k))
    ks = [c.src_k.get(l, c.src_k[any_l]) for l in range(s.src.num_layers)]
    vs = [c.src_v.get(l, c.src_v[any_l]) for l in range(s.src.num_layers)]
    return oracle.OracleProblem(s.src, s.dst, c.layer_map, c.wl.src_len, c.wl.tgt_seq_off, c.wl.s_max,
                                c.wl.t_max, ks, vs, c.w_k, c.w_v, c.wl.span_lo, c.wl.span_hi,
                                None if c.src_pos is None else c.src_pos.reshape(-1), c.tgt_pos,
                                form=s.form, k_layers=s.layers_per_target, low_rank=c.low_rank)


# Every comparison of the session: rel-L2, the literal max-abs and the count of elements above
# 3e-2, next to the test that made it (written out by conftest.py when KVX_PARITY_RECORD names
# a file, and summarised at the end of the run).
RECORD: List[dict] = []


def record(stats: dict, label: str = "") -> None:
    test = os.environ.get("PYTEST_CURRENT_TEST", "").split(" ")[0]
    RECORD.append(dict(stats, test=test, label=label))
    print(f"parity {test} {label}: rel_l2={stats['rel_l2']:.3e} max_abs={stats['max_abs']:.4e} "
          f"n_above_3e-2={stats['n_above_3e-2']} of {stats['n']}")


def compare(gpu: np.ndarray, ref: np.ndarray, dtype: str, label: str = "") -> dict:
    """Element-by-element comparison; records and returns stats, raises AssertionError on failure."""
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    assert gpu.shape == ref.shape, (gpu.shape, ref.shape)
    assert np.all(np.isfinite(gpu)), "non-finite output"
    err = np.abs(gpu - ref)
    nref = float(np.linalg.norm(ref))
    rel = float(np.linalg.norm(gpu - ref) / nref) if nref > 0 else float(np.linalg.norm(gpu - ref))
    stats = {"rel_l2": rel, "max_abs": float(err.max(initial=0.0)), "n": int(err.size),
             "n_above_3e-2": int((err > ABS_TOL).sum())}
    record(stats, label)
    assert rel <= REL_L2, stats
    if dtype == "bf16":
        bound = ABS_TOL + BF16_HALF_ULP_REL * np.abs(ref)
        bad = err > bound
        assert not bad.any(), dict(stats, n_bad=int(bad.sum()), worst=float((err - bound).max()))
    else:
        assert stats["max_abs"] <= ABS_TOL, stats
    return stats


def sample_rows(c: Case, n: int, seed: int = 0) -> List[tuple]:
    """(j, h, kv, tp) rows to check at full size: both ends of every sequence, tile
    boundaries and random rows, over all target layers and heads."""
    r = np.random.default_rng(seed)
    s = c.spec
    T = c.wl.total_tgt
    toks = set()
    for b in range(c.wl.batch):
        a, e = int(c.wl.tgt_seq_off[b]), int(c.wl.tgt_seq_off[b + 1])
        for t in (a, a + 1, e - 2, e - 1, a + 127, a + 128):
            if a <= t < e:
                toks.add(t)
    toks = sorted(toks)
    rows = []
    for i in range(n):
        j = int(r.integers(s.dst.num_layers)) if i >= s.dst.num_layers else i
        h = int(r.integers(s.dst.num_kv_heads))
        kv = int(r.integers(2))
        tp = toks[i % len(toks)] if i < 2 * len(toks) else int(r.integers(T))
        rows.append((j, h, kv, tp))
    return rows


def tokenization_workload(spec: synth.WorkloadSpec, n_bytes: Sequence[int], mean_src: float, mean_tgt: float,
                          key: int) -> synth.Workload:
    """A workload whose sequences are two independent tokenisations of byte strings of the given
    lengths (synth.draw_tokenizations), aligned by the oracle's builder: a finer target maps
    several target tokens to one source token, a coarser one gives long spans."""
    src_ends, tgt_ends = [], []
    for i, nb in enumerate(n_bytes):
        se, te = synth.draw_tokenizations(int(nb), mean_src, mean_tgt, key * 10 + i)
        src_ends.append(se)
        tgt_ends.append(te)
    so = np.concatenate([[0], np.cumsum([len(x) for x in src_ends])]).astype(np.int32)
    to = np.concatenate([[0], np.cumsum([len(x) for x in tgt_ends])]).astype(np.int32)
    se, te = np.concatenate(src_ends).astype(np.int32), np.concatenate(tgt_ends).astype(np.int32)
    lo, hi, n = oracle.build_alignment(so, se, to, te)
    assert n == 0
    src_len, tgt_len = np.diff(so).astype(np.int32), np.diff(to).astype(np.int32)
    return synth.Workload(spec, len(n_bytes), src_len, tgt_len, to, so, int(src_len.max()), int(tgt_len.max()),
                          lo, hi, se, te, None if spec.layer_map is None else np.array(spec.layer_map, np.int32))


def explicit_span_workload(spec: synth.WorkloadSpec, src_lens: Sequence[int], span_lo, span_hi) -> synth.Workload:
    """A workload with caller-chosen spans (packed over the sequences, indices within each),
    e.g. non-monotone or overlapping ones no tokenizer pair produces."""
    span_lo, span_hi = [np.asarray(x, np.int32) for x in span_lo], [np.asarray(x, np.int32) for x in span_hi]
    tgt_len = np.array([len(x) for x in span_lo], np.int32)
    src_len = np.array(src_lens, np.int32)
    to = np.concatenate([[0], np.cumsum(tgt_len)]).astype(np.int32)
    so = np.concatenate([[0], np.cumsum(src_len)]).astype(np.int32)
    return synth.Workload(spec, len(src_lens), src_len, tgt_len, to, so, int(src_len.max()), int(tgt_len.max()),
                          np.concatenate(span_lo), np.concatenate(span_hi), None, None,
                          None if spec.layer_map is None else np.array(spec.layer_map, np.int32))
