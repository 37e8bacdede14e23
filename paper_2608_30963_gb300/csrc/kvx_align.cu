// kvx_align.cu -- token-span alignment builder and RoPE table builder.
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

// One thread per target token.  Source token s belongs to the target token
// whose byte range [tgt_end[t-1], tgt_end[t]) holds its last byte src_end[s]-1,
// so target t's span starts at #{s : src_end[s] <= tgt_end[t-1]} and ends at
// #{s : src_end[s] <= tgt_end[t]}.  An empty span takes the source token that
// holds the target's last byte, which is the one at the span start.
__global__ void build_alignment_kernel(int batch, int total_tgt, const int* __restrict__ src_seq_off,
                                       const int* __restrict__ src_end, const int* __restrict__ tgt_seq_off,
                                       const int* __restrict__ tgt_end, int* __restrict__ span_lo,
                                       int* __restrict__ span_hi, unsigned* status)
{
    const int tp = blockIdx.x * blockDim.x + threadIdx.x;
    if (tp >= total_tgt) return;
    const int b = find_seq(tgt_seq_off, batch, tp);
    const int t = tp - __ldg(&tgt_seq_off[b]);
    const int s0 = __ldg(&src_seq_off[b]);
    const int S = __ldg(&src_seq_off[b + 1]) - s0;
    const int prev = t > 0 ? __ldg(&tgt_end[tp - 1]) : 0;
    const int cur = __ldg(&tgt_end[tp]);
    int lo = count_le(src_end + s0, S, prev);
    int hi = count_le(src_end + s0, S, cur);
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
    const int threads = 256;
    build_alignment_kernel<<<(total_tgt + threads - 1) / threads, threads, 0, stream>>>(
        batch, total_tgt, src_seq_off, src_end, tgt_seq_off, tgt_end, span_lo, span_hi, status);
    return cudaGetLastError();
}

}  // namespace kvx
