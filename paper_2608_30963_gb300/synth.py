"""Seeded synthetic workloads for cross-model KV translation.

This module only draws random numbers and lays them out; it holds none of the
translation's arithmetic (no RoPE, no projection, no span reduction), so both
the CUDA path and the CPU oracle can take their inputs from it.

Workloads follow the model pairs and context lengths of the paper's evaluation
(Section 6.1, Tables 3-5 and 7): Qwen2.5-7B -> Qwen2.5-1.5B, Qwen2.5-1.5B ->
Gemma-2-2B and Llama-3.1-70B -> Qwen2.5-7B KV geometries, plus a tiny fp32 pair
and a long-context batch sweep with a paged target cache.  The paper's datasets
(NoLiMa, LongBench2, FineWeb-Edu) are not used: synthetic K/V of the same
shapes stand in for the source caches they would produce.

Seeds: 0 source K/V, 1 W_K, 2 W_V, 3 outlier channels, 4 token alignment,
5 varlen lengths, 6 page permutation, 7 and 8 latent adapter factors.  Every stream is derived from
``numpy.random.SeedSequence([seed, *indices])`` so one layer can be
regenerated without drawing the others.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence

import numpy as np

SEED_KV, SEED_WK, SEED_WV, SEED_OUTLIER, SEED_ALIGN, SEED_VARLEN, SEED_PAGES, SEED_LATENT_A, SEED_LATENT_B = range(9)
FORM_GROUPED, FORM_DENSE = 0, 1


# ----------------------------------------------------------------------------
# bf16 storage format (IEEE binary32 truncated to its top 16 bits, RNE)
# ----------------------------------------------------------------------------
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (round to nearest even); return raw bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    nan = np.isnan(np.ascontiguousarray(x, dtype=np.float32))
    r = ((u >> 16) & 1) + 0x7FFF
    out = ((u + r) >> 16).astype(np.uint16)
    out[nan] = 0x7FC0
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def bf16_round(x: np.ndarray) -> np.ndarray:
    """float32 array whose values are exactly representable in bfloat16."""
    return bf16_bits_to_f32(f32_to_bf16_bits(x))


# ----------------------------------------------------------------------------
# geometry and workload description
# ----------------------------------------------------------------------------
ROPE_DEFAULT, ROPE_LINEAR, ROPE_LLAMA3 = 0, 1, 2


@dataclasses.dataclass(frozen=True)
class ModelGeom:
    num_layers: int
    num_kv_heads: int
    head_dim: int
    rope_base: float  # <= 0: the model applies no RoPE to K
    # RoPE frequency schedule: 0 plain, 1 linear position interpolation, 2 Llama-3.1
    rope_type: int = ROPE_DEFAULT
    rope_factor: float = 1.0
    rope_low_freq_factor: float = 1.0
    rope_high_freq_factor: float = 4.0
    rope_original_max_position: int = 8192
    rotary_dim: int = 0   # partial rotary: only the first rotary_dim channels rotate; 0 = all


@dataclasses.dataclass
class WorkloadSpec:
    name: str
    src: ModelGeom
    dst: ModelGeom
    dtype: str                      # "bf16" or "fp32"
    tgt_lens: Sequence[int]         # per-sequence target lengths
    cross_tokenizer: bool           # False: identity alignment (S_b == T_b)
    layer_map: Optional[Sequence[int]]  # None: nearest relative depth
    outliers: bool                  # 4 channels per (layer, K/V, head) scaled x8 before source RoPE
    paged: bool = False
    page_size: int = 16
    form: int = FORM_GROUPED        # which source heads feed a target head (grouped / dense)
    layers_per_target: int = 1      # source layers per target layer (layer_map is then [L_t, k])
    rank: int = 0                   # > 0: latent adapter factors instead of full matrices

    @property
    def heads_per_layer(self) -> int:
        """Source heads of one source layer in a target head's input row."""
        hs, ht = self.src.num_kv_heads, self.dst.num_kv_heads
        if self.form == FORM_DENSE:
            return hs
        return hs // ht if hs >= ht else 1

    @property
    def group_in(self) -> int:
        """Input width of one translator matrix: k source layers x heads x d_s."""
        return self.layers_per_target * self.heads_per_layer * self.src.head_dim


@dataclasses.dataclass
class Workload:
    spec: WorkloadSpec
    batch: int
    src_len: np.ndarray            # int32[B]
    tgt_len: np.ndarray            # int32[B]
    tgt_seq_off: np.ndarray        # int32[B+1]
    src_seq_off: np.ndarray        # int32[B+1] (packed source offsets, for byte ends)
    s_max: int
    t_max: int
    span_lo: Optional[np.ndarray]  # int32[T_total] within-sequence, None = identity
    span_hi: Optional[np.ndarray]
    src_end: Optional[np.ndarray]  # int32[S_total] byte-end offsets within each sequence
    tgt_end: Optional[np.ndarray]  # int32[T_total]
    layer_map: Optional[np.ndarray]  # explicit map or None
    page_table: Optional[np.ndarray] = None  # int32[B, max_pages]
    num_pages: int = 0
    max_pages: int = 0

    @property
    def total_tgt(self) -> int:
        return int(self.tgt_seq_off[-1])


def _rng(*key: int) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([int(k) for k in key]))


def _g(L, H, d, base):
    return ModelGeom(L, H, d, float(base))


QWEN7B = _g(28, 4, 128, 1e6)
QWEN1P5B = _g(28, 2, 128, 1e6)
GEMMA2B = _g(26, 4, 256, 1e4)
LLAMA70B = _g(80, 8, 128, 5e5)
# Llama-3.1's published RoPE schedule parameters (factor 8, low/high frequency factors 1 and 4,
# original context 8192); the 70B -> 7B workload keeps the plain schedule its description gives,
# this variant exercises the scaled one
LLAMA70B_SCALED = dataclasses.replace(LLAMA70B, rope_type=ROPE_LLAMA3, rope_factor=8.0,
                                      rope_low_freq_factor=1.0, rope_high_freq_factor=4.0,
                                      rope_original_max_position=8192)


def config_specs() -> Dict[str, WorkloadSpec]:
    specs = {
        "tiny_fp32": WorkloadSpec("tiny_fp32", _g(4, 2, 64, 1e4), _g(2, 1, 64, 1e4), "fp32",
                                  [256], False, [0, 2], False),
        "qwen7b_to_qwen1p5b_4k": WorkloadSpec("qwen7b_to_qwen1p5b_4k", QWEN7B, QWEN1P5B, "bf16",
                                              [4096], False, None, True),
        "llama70b_to_qwen7b_8k": WorkloadSpec("llama70b_to_qwen7b_8k", LLAMA70B, QWEN7B, "bf16",
                                              [8192], True, None, True),
    }
    # richer translator forms (the granularities the paper's Section 5 lists) on the
    # 70B -> 7B pair: one map per target layer over all source heads (in = 8 x 128), a group of
    # two source layers per target layer (in = 2 x 2 x 128), and a rank-64 latent adapter on
    # the 7B -> 1.5B pair
    specs["llama70b_to_qwen7b_8k_dense"] = WorkloadSpec(
        "llama70b_to_qwen7b_8k_dense", LLAMA70B, QWEN7B, "bf16", [8192], True, None, True, form=FORM_DENSE)
    specs["llama70b_to_qwen7b_8k_layers2"] = WorkloadSpec(
        "llama70b_to_qwen7b_8k_layers2", LLAMA70B, QWEN7B, "bf16", [8192], True, layer_groups(80, 28, 2), True,
        layers_per_target=2)
    specs["qwen7b_to_qwen1p5b_4k_latent64"] = WorkloadSpec(
        "qwen7b_to_qwen1p5b_4k_latent64", QWEN7B, QWEN1P5B, "bf16", [4096], False, None, True, rank=64)
    for t in (1024, 2048, 4096):
        n = f"qwen1p5b_to_gemma2b_{t // 1024}k"
        specs[n] = WorkloadSpec(n, QWEN1P5B, GEMMA2B, "bf16", [t], True, None, False)
    for L in (8192, 16384, 32768):
        for B in (1, 4, 8):
            n = f"longctx_{L // 1024}k_b{B}"
            lens = _varlen(L, B)
            specs[n] = WorkloadSpec(n, QWEN7B, QWEN1P5B, "bf16", lens, False, None, True, paged=True)
    return specs


def layer_groups(Ls: int, Lt: int, k: int) -> List[List[int]]:
    """A group of k consecutive source layers per target layer: target layer j takes the
    first k layers of the j-th of Lt equal contiguous slices of the Ls source layers
    (floor(j * Ls / Lt) onwards, clipped to the last layer).  A workload choice handed to
    both sides as an explicit layer map."""
    return [[min(Ls - 1, (j * Ls) // Lt + i) for i in range(k)] for j in range(Lt)]


def _varlen(L: int, B: int) -> List[int]:
    """Per-sequence lengths uniform in [ceil(L/2), L] (seed 5)."""
    r = _rng(SEED_VARLEN, L, B)
    return [int(x) for x in r.integers((L + 1) // 2, L + 1, size=B)]


# ----------------------------------------------------------------------------
# token alignment (cross-tokenizer) and byte offsets
# ----------------------------------------------------------------------------
SPAN_P = (0.75, 0.20, 0.05)  # P(span length = 1, 2, 3): mean 1.3


def draw_spans(T: int, b: int):
    """Monotone partition: target token t covers source tokens [lo[t], hi[t]).

    Also returns byte-end offsets of both tokenisations of one shared byte
    string: each source token is 1..6 bytes; a target token ends where its
    last source token ends.
    """
    r = _rng(SEED_ALIGN, b, T)
    lens = r.choice(np.array([1, 2, 3]), size=T, p=SPAN_P).astype(np.int64)
    hi = np.cumsum(lens)
    lo = hi - lens
    S = int(hi[-1]) if T else 0
    src_bytes = r.integers(1, 7, size=S)
    src_end = np.cumsum(src_bytes)
    tgt_end = src_end[hi - 1] if T else np.zeros(0, np.int64)
    return (lo.astype(np.int32), hi.astype(np.int32), S,
            src_end.astype(np.int32), tgt_end.astype(np.int32))


def draw_tokenizations(n_bytes: int, mean_src: float, mean_tgt: float, key: int):
    """Two independent tokenisations of the same n_bytes-byte string.

    Returns strictly increasing byte-end offsets (last = n_bytes) for each.  The
    target may be finer than the source, so some target tokens fall inside a
    single source token (the empty-span case of the alignment builder).
    """
    r = _rng(SEED_ALIGN, 1000 + key, n_bytes)

    def cut(mean):
        p = min(1.0, 1.0 / mean)
        ends = np.nonzero(r.random(n_bytes) < p)[0] + 1
        ends = ends[ends < n_bytes]
        return np.concatenate([ends, [n_bytes]]).astype(np.int32)

    return cut(mean_src), cut(mean_tgt)


# ----------------------------------------------------------------------------
# workload assembly
# ----------------------------------------------------------------------------
def make_workload(spec: WorkloadSpec, tgt_lens: Optional[Sequence[int]] = None) -> Workload:
    lens = list(tgt_lens if tgt_lens is not None else spec.tgt_lens)
    B = len(lens)
    tgt_len = np.array(lens, np.int32)
    tgt_seq_off = np.zeros(B + 1, np.int32)
    tgt_seq_off[1:] = np.cumsum(tgt_len)
    if spec.cross_tokenizer:
        los, his, S, se, te = [], [], [], [], []
        for b, T in enumerate(lens):
            lo, hi, s, src_end, tgt_end = draw_spans(T, b)
            los.append(lo); his.append(hi); S.append(s); se.append(src_end); te.append(tgt_end)
        src_len = np.array(S, np.int32)
        span_lo = np.concatenate(los).astype(np.int32)
        span_hi = np.concatenate(his).astype(np.int32)
        src_end = np.concatenate(se).astype(np.int32)
        tgt_end = np.concatenate(te).astype(np.int32)
    else:
        src_len = tgt_len.copy()
        span_lo = span_hi = src_end = tgt_end = None
    src_seq_off = np.zeros(B + 1, np.int32)
    src_seq_off[1:] = np.cumsum(src_len)
    wl = Workload(spec, B, src_len, tgt_len, tgt_seq_off, src_seq_off,
                  int(src_len.max()) if B else 0, int(tgt_len.max()) if B else 0,
                  span_lo, span_hi, src_end, tgt_end,
                  None if spec.layer_map is None else np.array(spec.layer_map, np.int32))
    if spec.paged:
        P = spec.page_size
        pages_per = [(int(t) + P - 1) // P for t in lens]
        wl.num_pages = int(sum(pages_per))
        wl.max_pages = max(pages_per) if pages_per else 0
        perm = _rng(SEED_PAGES, wl.num_pages).permutation(wl.num_pages).astype(np.int32)
        pt = np.full((B, max(wl.max_pages, 1)), -1, np.int32)
        k = 0
        for b, n in enumerate(pages_per):
            pt[b, :n] = perm[k:k + n]
            k += n
        wl.page_table = pt
    return wl


def source_kv(wl: Workload, layer: int, kv: int, pad_value: float = 0.0) -> np.ndarray:
    """Source K (kv=0, before the source RoPE) or V (kv=1) of one source layer.

    Layout [B, H_s, S_max, d_s] float32 holding values exactly representable in
    the workload's storage type.  N(0,1), plus (if the spec asks) 4 distinct
    channels per head scaled by 8.  Tokens past a sequence's length hold
    ``pad_value``.
    """
    g = wl.spec.src
    x = np.empty((wl.batch, g.num_kv_heads, wl.s_max, g.head_dim), np.float32)
    r = _rng(SEED_KV, layer, kv)
    for b in range(wl.batch):
        x[b] = r.standard_normal((g.num_kv_heads, wl.s_max, g.head_dim), dtype=np.float32)
    if wl.spec.outliers:
        ro = _rng(SEED_OUTLIER, layer, kv)
        for h in range(g.num_kv_heads):
            ch = ro.choice(g.head_dim, size=4, replace=False)
            x[:, h, :, ch] *= 8.0
    for b in range(wl.batch):
        x[b, :, int(wl.src_len[b]):, :] = pad_value
    return bf16_round(x) if wl.spec.dtype == "bf16" else x


def latent_factors(wl: Workload, kv: int):
    """Latent adapter factors of W_K (kv=0) / W_V (kv=1): A [L_t, H_t, in, rank] ~ N(0, 1/in)
    and B [L_t, H_t, rank, out] ~ N(0, 1/rank)."""
    s = wl.spec
    din, r, dout = s.group_in, s.rank, s.dst.head_dim
    ra = _rng(SEED_LATENT_A, kv, din, r)
    rb = _rng(SEED_LATENT_B, kv, r, dout)
    a = ra.standard_normal((s.dst.num_layers, s.dst.num_kv_heads, din, r), dtype=np.float32)
    b = rb.standard_normal((s.dst.num_layers, s.dst.num_kv_heads, r, dout), dtype=np.float32)
    a *= np.float32(1.0 / np.sqrt(din))
    b *= np.float32(1.0 / np.sqrt(r))
    if s.dtype == "bf16":
        a, b = bf16_round(a), bf16_round(b)
    return a, b


def weights(wl: Workload, kv: int) -> np.ndarray:
    """Translator matrices W_K (kv=0) / W_V (kv=1): [L_t, H_t, in, out] ~ N(0, 1/in)."""
    s = wl.spec
    din, dout = s.group_in, s.dst.head_dim
    r = _rng(SEED_WK if kv == 0 else SEED_WV, din, dout)
    w = np.empty((s.dst.num_layers, s.dst.num_kv_heads, din, dout), np.float32)
    for l in range(s.dst.num_layers):
        w[l] = r.standard_normal((s.dst.num_kv_heads, din, dout), dtype=np.float32)
    w *= np.float32(1.0 / np.sqrt(din))
    return bf16_round(w) if s.dtype == "bf16" else w
