// kvx_align.cu -- token-span alignment builder.
#include <climits>

#include "kvx_common.cuh"
#include "kvx_kernels.h"

namespace kvx {

// Number of entries of the increasing array a[0..n) that are <= x.
__device__ __forceinline__ int count_le(const int* a, int n, int x)
{
    int lo = 0, hi = n;
    while (lo < hi) {
        int mid = (lo + hi) >> 1;
        if (__ldg(&a[mid]) <= x) lo = mid + 1; else hi = mid;
    }
    return lo;
}

// Entries of the increasing window w[0..n) (n <= 64; entry j is register lo of lane j for j < 32,
// register hi of lane j-32 above) that are <= x: a fixed-step binary search over warp shuffles.
// Every lane of the warp must call it (each with its own x).
__device__ __forceinline__ int warp_count_le(int w_lo, int w_hi, int n, int x)
{
    int pos = 0;
#pragma unroll
    for (int step = 64; step > 0; step >>= 1) {
        const int cand = pos + step;                       // is entry cand-1 <= x ?
        const int j = cand - 1;
        const int a = __shfl_sync(0xffffffffu, w_lo, j & 31);
        const int c = __shfl_sync(0xffffffffu, w_hi, j & 31);
        const int v = cand <= n ? (j < 32 ? a : c) : INT_MAX;
        if (v <= x) pos = cand;
    }
    return pos;
}

// #{j : a[j] <= x} and #{j : a[j] <= y} for the increasing array a[0..n), found by the whole
// warp at once: each round the 32 lanes probe 32 points that split each bracket into 33 parts
// and a ballot keeps the part holding the answer, so a bracket of n shrinks to 32 in about
// log_33(n) rounds of one dependent load (3 for 5K tokens), instead of log_2(n) for one thread.
__device__ __forceinline__ int2 warp_count_le_global(const int* __restrict__ a, int n, int x, int y)
{
    const int lane = threadIdx.x & 31;
    int lx = 0, hx = n, ly = 0, hy = n;   // the answers lie in [l, h]
    while (hx - lx > 32 || hy - ly > 32) {
        const int sx = hx - lx, sy = hy - ly;
        // probe k tests "answer >= p_k" with p_k = l + (k+1) s / 33, i.e. a[p_k - 1] <= value
        const int px = lx + (int)((long long)(lane + 1) * sx / 33);
        const int py = ly + (int)((long long)(lane + 1) * sy / 33);
        const bool tx = sx > 32 && px > lx && __ldg(&a[px - 1]) <= x;
        const bool ty = sy > 32 && py > ly && __ldg(&a[py - 1]) <= y;
        const int cx = __popc(__ballot_sync(0xffffffffu, tx));
        const int cy = __popc(__ballot_sync(0xffffffffu, ty));
        if (sx > 32) {
            const int nl = cx > 0 ? lx + (int)((long long)cx * sx / 33) : lx;
            const int nh = cx < 32 ? lx + (int)((long long)(cx + 1) * sx / 33) - 1 : hx;
            lx = nl;
            hx = nh;
        }
        if (sy > 32) {
            const int nl = cy > 0 ? ly + (int)((long long)cy * sy / 33) : ly;
            const int nh = cy < 32 ? ly + (int)((long long)(cy + 1) * sy / 33) - 1 : hy;
            ly = nl;
            hy = nh;
        }
    }
    // brackets of at most 32 entries: the answer is l + #{j in [l, h) : a[j] <= value}
    const bool fx = lane < hx - lx && __ldg(&a[lx + lane]) <= x;
    const bool fy = lane < hy - ly && __ldg(&a[ly + lane]) <= y;
    return make_int2(lx + __popc(__ballot_sync(0xffffffffu, fx)), ly + __popc(__ballot_sync(0xffffffffu, fy)));
}

// Source token s belongs to the target token whose byte range [tgt_end[t-1], tgt_end[t]) holds
// its last byte src_end[s]-1, so target t's span starts at #{s : src_end[s] <= tgt_end[t-1]} and
// ends at #{s : src_end[s] <= tgt_end[t]}.  An empty span takes the source token that holds the
// target's last byte, which is the one at the span start.
//
// One warp per 32 consecutive target tokens.  When they all belong to one sequence (the common
// case), their spans are monotone, so one warp-wide search for the first lane's span start and
// the last lane's span end bounds the source tokens of the whole warp; if that window holds at
// most 64 tokens it is loaded into registers and every lane finds its two counts by shuffles.
// Otherwise each lane searches the global array itself.
__global__ void __launch_bounds__(128) build_alignment_kernel(int batch, int total_tgt,
                                                              const int* __restrict__ src_seq_off,
                                                              const int* __restrict__ src_end,
                                                              const int* __restrict__ tgt_seq_off,
                                                              const int* __restrict__ tgt_end,
                                                              int* __restrict__ span_lo, int* __restrict__ span_hi,
                                                              unsigned* status)
{
    const int lane = threadIdx.x & 31;
    const int tp0 = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5) * 32;
    if (tp0 >= total_tgt) return;                      // warp-uniform
    const int tp = tp0 + lane;
    const bool valid = tp < total_tgt;
    const int tpc = valid ? tp : total_tgt - 1;        // inactive lanes mirror the last token
    const int b = find_seq(tgt_seq_off, batch, tpc);
    const int t = tpc - __ldg(&tgt_seq_off[b]);
    const int s0 = __ldg(&src_seq_off[b]);
    const int S = __ldg(&src_seq_off[b + 1]) - s0;
    const int prev = t > 0 ? __ldg(&tgt_end[tpc - 1]) : 0;
    const int cur = __ldg(&tgt_end[tpc]);
    const int* se = src_end + s0;
    int lo, hi;
    const bool one_seq = __all_sync(0xffffffffu, b == __shfl_sync(0xffffffffu, b, 0));
    int w0 = 0, wn = 65;
    if (one_seq) {
        // window [w0, w0 + wn): source tokens at or after the first lane's span start and at or
        // before the last lane's span end
        const int2 c = warp_count_le_global(se, S, __shfl_sync(0xffffffffu, prev, 0), __shfl_sync(0xffffffffu, cur, 31));
        w0 = c.x;
        wn = c.y - c.x;
    }
    if (one_seq && wn >= 0 && wn <= 64) {
        const int e_lo = lane < wn ? __ldg(&se[w0 + lane]) : INT_MAX;
        const int e_hi = lane + 32 < wn ? __ldg(&se[w0 + lane + 32]) : INT_MAX;
        lo = w0 + warp_count_le(e_lo, e_hi, wn, prev);
        hi = w0 + warp_count_le(e_lo, e_hi, wn, cur);
    } else {
        lo = count_le(se, S, prev);
        hi = count_le(se, S, cur);
    }
    if (!valid) return;
    if (hi == lo) {
        hi = lo + 1;
        if (lo >= S) { lo = S - 1; hi = S; set_status(status, KVX_DEV_SPAN_CLAMPED); }
    }
    span_lo[tp] = lo;
    span_hi[tp] = hi;
}

cudaError_t launch_build_alignment(int batch, int total_tgt, const int* src_seq_off, const int* src_end,
                                   const int* tgt_seq_off, const int* tgt_end, int* span_lo, int* span_hi,
                                   unsigned* status, cudaStream_t stream)
{
    if (total_tgt <= 0) return cudaSuccess;
    const int threads = 128;   // 4 warps, one per 32 target tokens: many small blocks over the SMs
    build_alignment_kernel<<<(total_tgt + threads - 1) / threads, threads, 0, stream>>>(
        batch, total_tgt, src_seq_off, src_end, tgt_seq_off, tgt_end, span_lo, span_hi, status);
    return cudaGetLastError();
}

}  // namespace kvx
