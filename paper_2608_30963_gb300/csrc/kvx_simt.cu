// kvx_simt.cu -- CUDA-core translation kernel.
//
// One CTA per (32-token tile, target head, target layer, K|V).  Three phases:
//   1. gather the span rows of the source heads feeding the target head (its
//      GQA group, or every head in the dense form, of one or several source
//      layers), undo the source RoPE (K), take the span mean -> A[32][in]
//      (fp32, shared memory);
//   2. projection Y[32][d_t] = A . W[j,h] (fp32 FMA, W streamed from L2);
//   3. apply the target RoPE (K) and store the rows into the target cache.
// It serves the float32 caches and any geometry the tensor-core kernel does
// not take.  Paper: Section 5 (T_theta per layer and KV head).
#include "kvx_common.cuh"
#include "kvx_kernels.h"

namespace kvx {

constexpr int kSimtTile = 32;
constexpr int kSimtThreads = 256;

template <typename T>
__global__ void __launch_bounds__(kSimtThreads) translate_simt_kernel(const __grid_constant__ TranslateParams P)
{
    extern __shared__ float smem[];
    __shared__ TokenInfo tinfo[kSimtTile];
    float* A = smem;                              // [32][in]
    float* Y = smem + kSimtTile * P.in_dim;       // [32][dt]

    const int h = blockIdx.y;
    const int j = blockIdx.z >> 1;
    const int kv = blockIdx.z & 1;
    const int t0 = blockIdx.x * kSimtTile;
    const int ntok = min(kSimtTile, P.T_total - t0);
    if ((int)threadIdx.x < ntok) tinfo[threadIdx.x] = resolve_token(P, t0 + threadIdx.x);
    __syncthreads();

    const bool rot_s = kv == 0 && P.rs.enabled;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int hs = P.rhalf_s;   // rotating pairs (c, c + hs), c < hs; channels from 2 hs on do not rotate

    // ---- phase 1: un-rotate + span mean
    for (int tt = warp; tt < kSimtTile; tt += kSimtThreads / 32) {
        if (tt >= ntok) {
            for (int k = lane; k < P.in_dim; k += 32) A[tt * P.in_dim + k] = 0.f;
            continue;
        }
        const TokenInfo ti = tinfo[tt];
        for (int k = lane; k < P.in_dim; k += 32) {
            const int q = k / P.ds, c = k - q * P.ds;
            int slot, g;
            head_block(P, j, h, q, slot, g);
            const T* src = (const T*)(kv ? P.src_v[slot] : P.src_k[slot]);
            const T* base = src + (long long)ti.b * P.sb + (long long)g * P.sh;
            float acc = 0.f;
            for (int s = ti.lo; s < ti.hi; ++s) {
                const T* row = base + (long long)s * P.ss;
                float x = to_f32<T>(row[c]);
                if (rot_s && c < 2 * hs) {
                    const int i = c < hs ? c : c - hs;
                    const float xp = to_f32<T>(row[c < hs ? c + hs : c - hs]);
                    const float2 cs = rope_cs(P.rs, src_pos_of(P, ti.b, s), i);
                    // R(-theta): x_i' = x_i cos + x_{i+h} sin,  x_{i+h}' = x_{i+h} cos - x_i sin
                    x = c < hs ? fmaf(x, cs.x, xp * cs.y) : fmaf(x, cs.x, -xp * cs.y);
                }
                acc += x;
            }
            const int n = ti.hi - ti.lo;
            A[tt * P.in_dim + k] = n > 0 ? acc / (float)n : 0.f;
        }
    }
    __syncthreads();

    // ---- phase 2: projection, fp32 accumulate in ascending input index
    const T* W = (const T*)P.w + ((size_t)(kv * P.Lt + j) * P.Ht + h) * (size_t)P.in_dim * P.dt;
    const int G = kSimtThreads / P.dt;            // token groups (d_t <= 256)
    const int o = threadIdx.x % P.dt, grp = threadIdx.x / P.dt;
    for (int m0 = 0; m0 < kSimtTile / G; m0 += 8) {
        float acc[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) acc[u] = 0.f;
        for (int i = 0; i < P.in_dim; ++i) {
            const float w = to_f32<T>(W[(size_t)i * P.dt + o]);
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int tt = grp + G * (m0 + u);
                acc[u] = fmaf(A[tt * P.in_dim + i], w, acc[u]);
            }
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) Y[(grp + G * (m0 + u)) * P.dt + o] = acc[u];
    }
    __syncthreads();

    // ---- phase 3: target RoPE + store
    T* dst = (T*)(kv ? P.dst_v[j] : P.dst_k[j]);
    const bool rot_t = kv == 0 && P.rt.enabled;
    const int ht = P.rhalf_t;   // rotating pairs (c, c + ht), c < ht
    const long long hoff = dst_head_off(P, h);
    for (int idx = threadIdx.x; idx < ntok * P.dt; idx += kSimtThreads) {
        const int tt = idx / P.dt, c = idx - tt * P.dt;
        const TokenInfo& ti = tinfo[tt];
        if (ti.dst_off < 0) continue;
        float y = Y[tt * P.dt + c];
        if (rot_t && c < 2 * ht) {
            const int i = c < ht ? c : c - ht;
            const float yp = Y[tt * P.dt + (c < ht ? c + ht : c - ht)];
            const float2 cs = rope_cs(P.rt, ti.pt, i);
            // R(+theta): y_i' = y_i cos - y_{i+h} sin,  y_{i+h}' = y_{i+h} cos + y_i sin
            y = c < ht ? fmaf(y, cs.x, -yp * cs.y) : fmaf(y, cs.x, yp * cs.y);
        }
        dst[ti.dst_off + hoff + c] = from_f32<T>(y);
    }
}

// Latent adapter product W = A . B per (target layer, head, K|V), once at translator creation:
// A [n][in][rank], B [n][rank][out] -> W [n][in][out], fp32 accumulation over rank in ascending
// order, rounded to T.  One thread per output element.
template <typename T>
__global__ void fold_low_rank_kernel(const T* __restrict__ a, const T* __restrict__ b, T* __restrict__ w, int n,
                                     int in_dim, int rank, int out)
{
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    const long long per = (long long)in_dim * out;
    if (idx >= per * n) return;
    const int m = (int)(idx / per);
    const int rem = (int)(idx - (long long)m * per);
    const int i = rem / out, o = rem - i * out;
    const T* am = a + ((size_t)m * in_dim + i) * rank;
    const T* bm = b + (size_t)m * rank * out + o;
    float acc = 0.f;
    for (int c = 0; c < rank; ++c) acc = fmaf(to_f32<T>(am[c]), to_f32<T>(bm[(size_t)c * out]), acc);
    w[idx] = from_f32<T>(acc);
}

cudaError_t launch_fold_low_rank(const void* a, const void* b, void* w, int n, int in_dim, int rank, int out,
                                 int dtype, cudaStream_t stream)
{
    const long long total = (long long)n * in_dim * out;
    const unsigned blocks = (unsigned)((total + 255) / 256);
    if (dtype == KVX_BF16)
        fold_low_rank_kernel<__nv_bfloat16><<<blocks, 256, 0, stream>>>(
            (const __nv_bfloat16*)a, (const __nv_bfloat16*)b, (__nv_bfloat16*)w, n, in_dim, rank, out);
    else
        fold_low_rank_kernel<float><<<blocks, 256, 0, stream>>>((const float*)a, (const float*)b, (float*)w, n,
                                                                 in_dim, rank, out);
    return cudaGetLastError();
}

size_t simt_smem_bytes(int in_dim, int dt)
{
    return (size_t)kSimtTile * (in_dim + dt) * sizeof(float);
}

cudaError_t launch_translate_simt(const TranslateParams& P, int dtype, cudaStream_t stream)
{
    const size_t smem = simt_smem_bytes(P.in_dim, P.dt);
    dim3 grid((P.T_total + kSimtTile - 1) / kSimtTile, P.Ht, P.Lt * 2);
    cudaError_t err;
    if (dtype == KVX_BF16) {
        err = cudaFuncSetAttribute(translate_simt_kernel<__nv_bfloat16>,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
        translate_simt_kernel<__nv_bfloat16><<<grid, kSimtThreads, smem, stream>>>(P);
    } else {
        err = cudaFuncSetAttribute(translate_simt_kernel<float>,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
        translate_simt_kernel<float><<<grid, kSimtThreads, smem, stream>>>(P);
    }
    return cudaGetLastError();
}

}  // namespace kvx
