// kvx_common.cuh -- shared definitions of the kvx CUDA kernels (library-internal).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/kvx.h"

namespace kvx {

constexpr int KVX_MAX_ALIGNED_LAYERS = 96;   // target layers the identity-alignment kernel takes (param space)
constexpr int KVX_MAX_SRC_SLOTS = 256;       // (target layer, source-layer slot) pairs one launch addresses
constexpr int KVX_MAX_ALIGNED_BATCH = 256;   // sequences whose metadata it keeps in shared memory

// Rotation frequencies as fixed-point turns: turns[i] = 2^64 * f_i / (2 pi), evaluated in
// double and converted to an integer by truncation, f_i = base^(-2i/d) (on the host).  For an
// integer position p, p * turns[i] mod 2^64 is the fractional part of the angle p * f_i in
// turns, exact up to the rounding of turns[i] (|error| <= p * 2^-52 turn), so the range
// reduction costs one 64-bit multiply and no table of angles.
struct RopeTable {
    const unsigned long long* turns;   // device [d/2]; entries of pairs that do not rotate are 0
    int half;                          // d/2
    int enabled;                       // 0: no rotation
};

// Channels of K that rotate (the first ones; all of them unless the head is partial rotary).
__host__ __device__ inline int rope_rot_dim(const kvx_model_geom& g)
{
    return g.rotary_dim > 0 ? g.rotary_dim : g.head_dim;
}

// Kernels that pair element k of the first half of a head row with element k + d/2 walk
// "pair slots" k < d/2.  A partial rotary head pairs channel i with i + rhalf (i < rhalf)
// and leaves the channels from 2 rhalf on alone, so slot k covers the two channels
//   (k, k + rhalf)       for k < rhalf  (a rotating pair), else
//   (k + rhalf, k + d/2)                (two channels that do not rotate),
// every channel exactly once; with rhalf = d/2 this is (k, k + d/2).  rhalf is a multiple
// of 8, so a chunk of 8 (or 4) slots maps to two runs of consecutive channels.
__host__ __device__ __forceinline__ void pair_channels(int k, int half, int rhalf, int& lo, int& hi)
{
    if (k < rhalf) { lo = k; hi = k + rhalf; }
    else { lo = k + rhalf; hi = k + half; }
}

// Rotation frequency f_i of channel pair (i, i + n/2), n = rope_rot_dim, under the model's schedule
// (kvx_rope_type in kvx.h), in double.  Host code turns it into fixed-point turns
// once per translator; the allocation-free entry point does the same on the device.
__host__ __device__ inline double rope_inv_freq(const kvx_model_geom& g, int i)
{
    const double f = pow(g.rope_base, -2.0 * (double)i / (double)rope_rot_dim(g));
    if (g.rope_type == KVX_ROPE_LINEAR) return f / g.rope_factor;
    if (g.rope_type != KVX_ROPE_LLAMA3) return f;
    const double wavelen = 6.283185307179586 / f;
    const double orig = (double)g.rope_original_max_position;
    if (wavelen < orig / g.rope_high_freq_factor) return f;            // high-frequency band: kept
    if (wavelen > orig / g.rope_low_freq_factor) return f / g.rope_factor;   // low band: interpolated
    const double m = (orig / wavelen - g.rope_low_freq_factor) / (g.rope_high_freq_factor - g.rope_low_freq_factor);
    return (1.0 - m) * (f / g.rope_factor) + m * f;
}

// Schedule parameters valid for the model's rope_type (host-side validation).
inline bool rope_schedule_ok(const kvx_model_geom& g)
{
    if (g.rotary_dim != 0 && (g.rotary_dim < 16 || g.rotary_dim > g.head_dim || g.rotary_dim % 16)) return false;
    if (g.rope_base <= 0.0) return g.rope_type >= KVX_ROPE_DEFAULT && g.rope_type <= KVX_ROPE_LLAMA3;
    switch (g.rope_type) {
    case KVX_ROPE_DEFAULT: return true;
    case KVX_ROPE_LINEAR: return g.rope_factor > 0.0;
    case KVX_ROPE_LLAMA3:
        return g.rope_factor > 0.0 && g.rope_low_freq_factor > 0.0 &&
               g.rope_high_freq_factor > g.rope_low_freq_factor && g.rope_original_max_position > 0;
    default: return false;
    }
}

// Everything one kvx_translate launch needs, passed by value (graph-capturable;
// no per-call device allocation or copy).
struct TranslateParams {
    // geometry
    int Hs, ds, Ht, dt;
    int in_dim;     // input width of one translator matrix
    int r;          // source heads grouped into one target head (Hs >= Ht), else 1
    int e;          // target heads sharing one source head (Ht > Hs), else 1
    int dense;      // 1: every source KV head feeds each target head (per-layer form)
    int kl;         // source layers concatenated into one target layer's input (group of layers)
    int hpl;        // source heads per source layer in one input row: in_dim = kl * hpl * ds
    int Lt;
    // source cache
    int batch, src_max_seq;
    long long sb, sh, ss;
    const int* src_seq_len;
    const int* src_pos;
    // target tokens
    int T_total;
    const int* seq_off;
    const int* span_lo;
    const int* span_hi;
    const int* tgt_pos;
    // target cache
    int paged, dst_max_seq;
    long long db, dh, dts;
    const int* page_table;
    int max_pages, page_size, num_pages;
    // rotation
    RopeTable rs, rt;
    int rhalf_s, rhalf_t;   // rotating pairs (i, i + rhalf), i < rhalf, of the source / target head:
                            // rotary_dim/2 (= d/2 unless the head is partial rotary)
    int rope_same;   // source and target rotations coincide (same head_dim, same frequencies)
    int max_position;
    int plain_stores;   // write target rows with 16-byte stores from the threads instead of the bulk-copy
                        // unit (destinations on another device, reached over the peer mapping)
    // diagnostics of the bounded waits (kvx_debug_stall_next_translate): 0 = off
    unsigned long long wait_ns;   // bound of each on-chip wait instead of ~1 s
    int stall_unit1;              // identity kernel: CTA 0's producer issues no copies from its
                                  // (stall_unit1 - 1)-th unit on, so the waits for them run out
    unsigned* status;
    // weights (layout depends on the kernel)
    const void* w;
    // source K/V per (target layer j, layer slot k) at [j * kl + k], and the target layer's K/V
    const void* src_k[KVX_MAX_SRC_SLOTS];
    const void* src_v[KVX_MAX_SRC_SLOTS];
    void* dst_k[KVX_MAX_TARGET_LAYERS];
    void* dst_v[KVX_MAX_TARGET_LAYERS];
};

// Validated translator geometry (host side), shared by kvx_translator_create and the fitter.
struct Geometry {
    kvx_translator_desc desc;            // the caller's description, layer_map pointer cleared
    int layer_map[KVX_MAX_SRC_SLOTS];    // [j * kl + k]: source layers of target layer j
    int in_dim, r, e, dense, kl, hpl;
    int max_position;
    unsigned long long turns[256];       // fixed-point turns: source [ds/2] | target [dt/2]
    int rope_same;                       // source and target turns identical
};
// Checks a description and derives the geometry; no CUDA call.  On failure returns the status
// and writes a message (prefixed with who) to err[512].
kvx_status make_geometry(const kvx_translator_desc* desc, const char* who, Geometry& g, char* err);
// Launch parameters of one call over the caller's caches (argument checks included).
kvx_status make_params(const Geometry& g, const unsigned long long* dev_turns, unsigned* status, const void* w,
                       const kvx_src_kv* src, const kvx_tgt_tokens* tgt, const kvx_dst_kv* dst, TranslateParams& P,
                       const char* who, char* err);
// Thread-local message returned by kvx_last_error().
void set_last_error(const char* msg);

// Target heads that read the same input rows: the e heads of a GQA expansion group, every head
// in the dense per-layer form, else 1.
__host__ __device__ inline int share_heads(int dense, int r, int e, int Ht) { return dense ? Ht : (r == 1 ? e : 1); }
__host__ __device__ inline int share_heads(const TranslateParams& P) { return share_heads(P.dense, P.r, P.e, P.Ht); }

// First source head feeding target head h: its GQA group (h*r), the source head it
// repeats (h/e), or head 0 in the dense per-layer form.
__device__ __forceinline__ int src_head0(const TranslateParams& P, int h)
{
    return P.dense ? 0 : (P.r > 1 ? h * P.r : h / P.e);
}

// Head-block q of target head h's input row (d_s channels of one source head):
// the source cache slot (index into src_k / src_v) and the source head.
__device__ __forceinline__ void head_block(const TranslateParams& P, int j, int h, int q, int& slot, int& g)
{
    const int k = q / P.hpl;
    slot = j * P.kl + k;
    g = src_head0(P, h) + (q - k * P.hpl);
}

__device__ __forceinline__ void set_status(unsigned* status, unsigned bit)
{
    if (status) atomicOr(status, bit);
}

// (cos, sin) of the angle whose turns are p * G (mod 1): the top 32 bits of the
// 64-bit product are the signed fraction of a turn in [-1/2, 1/2), i.e. an
// angle in [-pi, pi) where the hardware sine/cosine is accurate to ~4e-7.
__device__ __forceinline__ float2 turn_cs(unsigned long long G, int p)
{
    const unsigned long long t = G * (unsigned long long)(unsigned)p;
    const float a = (float)(int)(t >> 32) * 1.4629180792671596e-09f;   // 2 pi / 2^32
    float sn, cs;
    __sincosf(a, &sn, &cs);
    return make_float2(cs, sn);
}

__device__ __forceinline__ float2 rope_cs(const RopeTable& t, int p, int i)
{
    return turn_cs(__ldg(&t.turns[i]), p);
}

__device__ __forceinline__ int clamp_pos(int p, int max_position, unsigned* status)
{
    if (p < 0 || p >= max_position) {
        set_status(status, KVX_DEV_POS_CLAMPED);
        p = p < 0 ? 0 : max_position - 1;
    }
    return p;
}

// Sequence holding packed target token tp (seq_off non-decreasing; empty sequences skipped).
__device__ __forceinline__ int find_seq(const int* seq_off, int batch, int tp)
{
    int lo = 0, hi = batch - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (__ldg(&seq_off[mid]) <= tp) lo = mid; else hi = mid - 1;
    }
    return lo;
}

template <typename T> __device__ __forceinline__ float to_f32(T x);
template <> __device__ __forceinline__ float to_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T> __device__ __forceinline__ T from_f32(float x);
template <> __device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) { return __float2bfloat16_rn(x); }

// Per-target-token information resolved once per tile.
struct TokenInfo {
    int b;        // sequence
    int t;        // index within the sequence
    int lo, hi;   // clamped source span (within sequence), hi > lo unless the source is empty
    int pt;       // target RoPE position (clamped)
    long long dst_off;  // element offset of the output row for head 0 in the target cache, -1 = skip
};

__device__ __forceinline__ TokenInfo resolve_token(const TranslateParams& P, int tp)
{
    TokenInfo ti;
    ti.b = find_seq(P.seq_off, P.batch, tp);
    ti.t = tp - __ldg(&P.seq_off[ti.b]);
    int S = __ldg(&P.src_seq_len[ti.b]);
    if (S > P.src_max_seq || S < 0) { set_status(P.status, KVX_DEV_SEQ_CLAMPED); S = S < 0 ? 0 : P.src_max_seq; }
    int lo, hi;
    if (P.span_lo) { lo = __ldg(&P.span_lo[tp]); hi = __ldg(&P.span_hi[tp]); }
    else { lo = ti.t; hi = ti.t + 1; }
    if (lo < 0 || hi > S || hi <= lo) {
        set_status(P.status, KVX_DEV_SPAN_CLAMPED);
        lo = lo < 0 ? 0 : (lo > S - 1 ? S - 1 : lo);
        hi = hi > S ? S : hi;
        if (hi <= lo) hi = lo + 1;
        if (S == 0) { lo = 0; hi = 0; }
    }
    ti.lo = lo; ti.hi = hi;
    int p = P.tgt_pos ? __ldg(&P.tgt_pos[tp]) : ti.t;
    ti.pt = P.rt.enabled ? clamp_pos(p, P.max_position, P.status) : 0;
    if (!P.paged) {
        if (ti.t >= P.dst_max_seq) { set_status(P.status, KVX_DEV_SEQ_CLAMPED); ti.dst_off = -1; }
        else ti.dst_off = (long long)ti.b * P.db + (long long)ti.t * P.dts;
    } else {
        int pi = ti.t / P.page_size;
        int page = pi < P.max_pages ? __ldg(&P.page_table[(size_t)ti.b * P.max_pages + pi]) : -1;
        if (page < 0 || page >= P.num_pages) { set_status(P.status, KVX_DEV_PAGE_INVALID); ti.dst_off = -1; }
        else ti.dst_off = ((long long)page * P.page_size + (ti.t % P.page_size)) * (long long)P.Ht * P.dt;
    }
    return ti;
}

// Element offset of head h within an output row block.
__device__ __forceinline__ long long dst_head_off(const TranslateParams& P, int h)
{
    return P.paged ? (long long)h * P.dt : (long long)h * P.dh;
}

__device__ __forceinline__ int src_pos_of_seq(const int* src_pos, int src_max_seq, int b, int s, int max_position,
                                              unsigned* status)
{
    const int p = src_pos ? __ldg(&src_pos[(size_t)b * src_max_seq + s]) : s;
    return clamp_pos(p, max_position, status);
}

__device__ __forceinline__ int src_pos_of(const TranslateParams& P, int b, int s)
{
    int p = P.src_pos ? __ldg(&P.src_pos[(size_t)b * P.src_max_seq + s]) : s;
    return clamp_pos(p, P.max_position, P.status);
}

}  // namespace kvx
