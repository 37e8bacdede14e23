// kvx_fit.cu -- closed-form fit of the linear translator (paper Section 5).
//
// Section 5 gives the learning objective L_KV = D(T_theta(KV_A(C)), KV_B(C)).  With D the
// squared Euclidean distance over target tokens plus a ridge term lambda |W|^2, every
// (target layer j, target head h, K|V) group is a least-squares problem solved by the normal
// equations (X^T X + lambda I) W = X^T Y:
//   X rows: the translator's input rows (span mean of the un-rotated source rows, as the
//           translation forms them), rounded to the cache dtype;
//   Y rows: the target model's own cache rows, target RoPE undone for K.
// Three steps:
//   1. fit_rows_kernel builds X and Y for one pass of up to chunk tokens, every group at once
//      (HBM-bound gather, CUDA cores);
//   2. two strided-batched cuBLAS GEMMs over the groups add X^T X and X^T Y into fp32 sums
//      (a plain dense contraction over tokens: tensor cores through the library);
//   3. at solve time, one CTA per group factors X^T X + lambda I = L L^T and runs the two
//      triangular solves per output column: fit_solve_small_kernel in fp32 shared memory for
//      in <= 256, fit_solve_kernel in double global memory above.
#include <cublas_v2.h>
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include "kvx_common.cuh"
#include "kvx_kernels.h"

namespace kvx {
namespace {

constexpr int kFitTile = 32;
constexpr int kFitThreads = 256;
constexpr int kSolveThreads = 256;
constexpr unsigned kFitNotPosDef = 0x20u;   // status bit: a system was not positive definite

struct FitRows {
    void* x;      // [groups][chunk][in]
    void* y;      // [groups][chunk][dt]
    int chunk;    // token capacity of one group's block
    int t0;       // first packed target token of this pass
    int n;        // tokens in this pass
};

// 16-byte chunks of T: VEC elements, as raw words and back.
template <typename T> struct Chunk;
template <> struct Chunk<__nv_bfloat16> {
    static constexpr int VEC = 8;
    __device__ static void unpack(const uint4& w, float (&x)[8])
    {
        const uint32_t v[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) { x[2 * i] = __uint_as_float(v[i] << 16); x[2 * i + 1] = __uint_as_float(v[i] & 0xFFFF0000u); }
    }
    __device__ static uint4 pack(const float (&x)[8])
    {
        uint32_t v[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            __nv_bfloat162 b = __floats2bfloat162_rn(x[2 * i], x[2 * i + 1]);
            v[i] = *reinterpret_cast<uint32_t*>(&b);
        }
        return make_uint4(v[0], v[1], v[2], v[3]);
    }
};
template <> struct Chunk<float> {
    static constexpr int VEC = 4;
    __device__ static void unpack(const uint4& w, float (&x)[4])
    {
        x[0] = __uint_as_float(w.x); x[1] = __uint_as_float(w.y); x[2] = __uint_as_float(w.z); x[3] = __uint_as_float(w.w);
    }
    __device__ static uint4 pack(const float (&x)[4])
    {
        return make_uint4(__float_as_uint(x[0]), __float_as_uint(x[1]), __float_as_uint(x[2]), __float_as_uint(x[3]));
    }
};

// One CTA per (32-token tile of the pass, target head, target layer * 2 + K|V).  A work item is
// one chunk pair: VEC pair slots [c, c+VEC) of one head row, i.e. channels [c, c+VEC) and their
// rotary partners [c+d/2, ...) (pair_channels for partial rotary heads), read and written as
// 16-byte words, with one (cos, sin) per rotating pair.
// X items: (token, head-block q, chunk pair); Y items: (token, chunk pair).
template <typename T>
__global__ void __launch_bounds__(kFitThreads) fit_rows_kernel(const __grid_constant__ TranslateParams P, const FitRows R)
{
    constexpr int VEC = Chunk<T>::VEC;
    __shared__ TokenInfo tinfo[kFitTile];
    const int h = blockIdx.y;
    const int j = blockIdx.z >> 1;
    const int kv = blockIdx.z & 1;
    const int g = (j * P.Ht + h) * 2 + kv;
    const int tt0 = blockIdx.x * kFitTile;
    const int ntok = min(kFitTile, R.n - tt0);
    if ((int)threadIdx.x < ntok) tinfo[threadIdx.x] = resolve_token(P, R.t0 + tt0 + (int)threadIdx.x);
    __syncthreads();

    T* X = (T*)R.x + ((size_t)g * R.chunk + tt0) * P.in_dim;
    T* Y = (T*)R.y + ((size_t)g * R.chunk + tt0) * P.dt;
    const T* tgt = (const T*)(kv ? P.dst_v[j] : P.dst_k[j]);
    const long long hoff = dst_head_off(P, h);
    const bool rot_s = kv == 0 && P.rs.enabled;
    const bool rot_t = kv == 0 && P.rt.enabled;
    const int hs = P.ds >> 1, ht = P.dt >> 1;
    const int ncp_s = hs / VEC, ncp_t = ht / VEC;       // chunk pairs per head row
    const int heads = P.in_dim / P.ds;                  // head-blocks in an input row
    const int x_items = ntok * heads * ncp_s;
    for (int it = threadIdx.x; it < x_items; it += blockDim.x) {
        const int tt = it / (heads * ncp_s);
        const int rem = it - tt * (heads * ncp_s);
        const int q = rem / ncp_s, cp = rem - q * ncp_s;
        const TokenInfo ti = tinfo[tt];
        int c_lo, c_hi;
        pair_channels(cp * VEC, hs, P.rhalf_s, c_lo, c_hi);
        float a0[VEC], a1[VEC];
#pragma unroll
        for (int e = 0; e < VEC; ++e) { a0[e] = 0.f; a1[e] = 0.f; }
        if (ti.dst_off >= 0 && ti.hi > ti.lo) {
            int slot, gs;
            head_block(P, j, h, q, slot, gs);
            const T* base = (const T*)(kv ? P.src_v[slot] : P.src_k[slot]) + (long long)ti.b * P.sb +
                            (long long)gs * P.sh;
            for (int s = ti.lo; s < ti.hi; ++s) {
                const T* row = base + (long long)s * P.ss;
                float x0[VEC], x1[VEC];
                Chunk<T>::unpack(__ldg(reinterpret_cast<const uint4*>(row + c_lo)), x0);
                Chunk<T>::unpack(__ldg(reinterpret_cast<const uint4*>(row + c_hi)), x1);
                if (rot_s && cp * VEC < P.rhalf_s) {
                    const int pos = src_pos_of(P, ti.b, s);
#pragma unroll
                    for (int e = 0; e < VEC; ++e) {   // R(-theta)
                        const float2 cs = rope_cs(P.rs, pos, cp * VEC + e);
                        a0[e] += fmaf(x0[e], cs.x, x1[e] * cs.y);
                        a1[e] += fmaf(x1[e], cs.x, -x0[e] * cs.y);
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < VEC; ++e) { a0[e] += x0[e]; a1[e] += x1[e]; }
                }
            }
            const float inv = 1.f / (float)(ti.hi - ti.lo);
#pragma unroll
            for (int e = 0; e < VEC; ++e) { a0[e] *= inv; a1[e] *= inv; }
        }
        T* xr = X + (size_t)tt * P.in_dim + q * P.ds;
        *reinterpret_cast<uint4*>(xr + c_lo) = Chunk<T>::pack(a0);
        *reinterpret_cast<uint4*>(xr + c_hi) = Chunk<T>::pack(a1);
    }
    const int y_items = ntok * ncp_t;
    for (int it = threadIdx.x; it < y_items; it += blockDim.x) {
        const int tt = it / ncp_t, cp = it - tt * ncp_t;
        const TokenInfo ti = tinfo[tt];
        int c_lo, c_hi;
        pair_channels(cp * VEC, ht, P.rhalf_t, c_lo, c_hi);
        float y0[VEC], y1[VEC];
        if (ti.dst_off >= 0 && ti.hi > ti.lo) {
            const T* row = tgt + ti.dst_off + hoff;
            Chunk<T>::unpack(__ldg(reinterpret_cast<const uint4*>(row + c_lo)), y0);
            Chunk<T>::unpack(__ldg(reinterpret_cast<const uint4*>(row + c_hi)), y1);
            if (rot_t && cp * VEC < P.rhalf_t) {
#pragma unroll
                for (int e = 0; e < VEC; ++e) {   // R(-theta)
                    const float2 cs = rope_cs(P.rt, ti.pt, cp * VEC + e);
                    const float u0 = fmaf(y0[e], cs.x, y1[e] * cs.y), u1 = fmaf(y1[e], cs.x, -y0[e] * cs.y);
                    y0[e] = u0;
                    y1[e] = u1;
                }
            }
        } else {
#pragma unroll
            for (int e = 0; e < VEC; ++e) { y0[e] = 0.f; y1[e] = 0.f; }
        }
        T* yr = Y + (size_t)tt * P.dt;
        *reinterpret_cast<uint4*>(yr + c_lo) = Chunk<T>::pack(y0);
        *reinterpret_cast<uint4*>(yr + c_hi) = Chunk<T>::pack(y1);
    }
}

// One CTA per group g = (j*Ht + h)*2 + kv.  G: fp32 X^T X [in][in]; C: fp32 X^T Y, column-major
// [dt][in] (element (a, o) at o*in + a); A, Z: double scratch [in][in] and [in][dt].
// W out: the group's [in][dt] block of W_K or W_V in the cache dtype.
template <typename T>
__global__ void __launch_bounds__(kSolveThreads) fit_solve_kernel(const float* __restrict__ G,
                                                                  const float* __restrict__ C, double* A, double* Z,
                                                                  T* wk, T* wv, int in, int dt, double lambda,
                                                                  unsigned* status)
{
    __shared__ int bad;
    const int g = blockIdx.x;
    double* a = A + (size_t)g * in * in;
    double* z = Z + (size_t)g * in * dt;
    const float* gg = G + (size_t)g * in * in;
    const float* cc = C + (size_t)g * in * dt;
    if (threadIdx.x == 0) bad = 0;
    for (int i = threadIdx.x; i < in * in; i += blockDim.x) {
        const int r = i / in, c = i - r * in;
        a[i] = c <= r ? (double)gg[i] + (r == c ? lambda : 0.0) : 0.0;
    }
    __syncthreads();
    // right-looking Cholesky on the lower triangle: a = L L^T
    for (int k = 0; k < in; ++k) {
        if (threadIdx.x == 0) {
            double d = a[(size_t)k * in + k];
            if (!(d > 0.0)) { bad = 1; d = 1.0; }
            a[(size_t)k * in + k] = sqrt(d);
        }
        __syncthreads();
        const double dk = a[(size_t)k * in + k];
        for (int r = k + 1 + threadIdx.x; r < in; r += blockDim.x) a[(size_t)r * in + k] /= dk;
        __syncthreads();
        const int m = in - k - 1;
        for (int idx = threadIdx.x; idx < m * m; idx += blockDim.x) {
            const int rr = k + 1 + idx / m, c2 = k + 1 + idx % m;
            if (c2 <= rr) a[(size_t)rr * in + c2] -= a[(size_t)rr * in + k] * a[(size_t)c2 * in + k];
        }
        __syncthreads();
    }
    // per output column o: L u = c (forward), L^T w = u (backward); z holds u then w, [in][dt]
    for (int o = threadIdx.x; o < dt; o += blockDim.x) {
        for (int r = 0; r < in; ++r) {
            double v = (double)cc[(size_t)o * in + r];
            for (int k = 0; k < r; ++k) v -= a[(size_t)r * in + k] * z[(size_t)k * dt + o];
            z[(size_t)r * dt + o] = v / a[(size_t)r * in + r];
        }
        for (int r = in - 1; r >= 0; --r) {
            double v = z[(size_t)r * dt + o];
            for (int k = r + 1; k < in; ++k) v -= a[(size_t)k * in + r] * z[(size_t)k * dt + o];
            z[(size_t)r * dt + o] = v / a[(size_t)r * in + r];
        }
    }
    __syncthreads();
    T* w = (g & 1) ? wv : wk;
    const size_t off = (size_t)(g >> 1) * in * dt;   // (j*Ht + h) block of [Lt][Ht][in][dt]
    for (int i = threadIdx.x; i < in * dt; i += blockDim.x) w[off + i] = from_f32<T>(bad ? 0.f : (float)z[i]);
    if (bad && threadIdx.x == 0) set_status(status, kFitNotPosDef);
}

// in <= kSmallSolve: the factor lives in shared memory as fp32, packed lower triangle (row r at
// r(r+1)/2), followed by `cols` columns of solutions [in][cols].  The sums X^T X are fp32 already,
// so a float factorisation loses nothing against them; it removes the L2 round trips of the
// double, global-memory kernel above.  One CTA per group.
constexpr int kSmallSolve = 256;
constexpr int kSmallSolveThreads = 512;
constexpr int kSmallSolveSmem = 227 * 1024 - 2048;   // dynamic shared memory budget

template <typename T>
__global__ void __launch_bounds__(kSmallSolveThreads) fit_solve_small_kernel(const float* __restrict__ G,
                                                                             const float* __restrict__ C, T* wk,
                                                                             T* wv, int in, int dt, int cols,
                                                                             float lambda, unsigned* status)
{
    extern __shared__ float Lp[];          // packed lower triangle, then the solution block
    __shared__ float colk[kSmallSolve];    // column k of L below the diagonal
    __shared__ int bad;
    const int g = blockIdx.x;
    const float* gg = G + (size_t)g * in * in;
    const float* cc = C + (size_t)g * in * dt;
    auto at = [](int r, int c) { return r * (r + 1) / 2 + c; };
    float* zs = Lp + at(in, 0);            // [in][cols]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
    if (threadIdx.x == 0) bad = 0;
    for (int r = warp; r < in; r += nwarps)
        for (int c = lane; c <= r; c += 32) Lp[at(r, c)] = gg[(size_t)r * in + c] + (r == c ? lambda : 0.f);
    __syncthreads();
    // right-looking Cholesky: Lp = L with L L^T = X^T X + lambda I
    for (int k = 0; k < in; ++k) {
        if (threadIdx.x == 0) {
            float d = Lp[at(k, k)];
            if (!(d > 0.f)) { bad = 1; d = 1.f; }
            Lp[at(k, k)] = sqrtf(d);
        }
        __syncthreads();
        const float dk = Lp[at(k, k)];
        for (int r = k + 1 + threadIdx.x; r < in; r += blockDim.x) {
            const float v = Lp[at(r, k)] / dk;
            Lp[at(r, k)] = v;
            colk[r] = v;
        }
        __syncthreads();
        for (int r = k + 1 + warp; r < in; r += nwarps) {
            const float lr = colk[r];
            for (int c = k + 1 + lane; c <= r; c += 32) Lp[at(r, c)] -= lr * colk[c];
        }
        __syncthreads();
    }
    T* w = (g & 1) ? wv : wk;
    const size_t off = (size_t)(g >> 1) * in * dt;
    for (int o0 = 0; o0 < dt; o0 += cols) {
        const int nc = min(cols, dt - o0);
        // one thread per output column: L u = c, then L^T w = u, four independent partial sums
        for (int o = threadIdx.x; o < nc; o += blockDim.x) {
            for (int r = 0; r < in; ++r) {
                const float* lr = Lp + at(r, 0);
                float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
                int k = 0;
                for (; k + 3 < r; k += 4) {
                    s0 = fmaf(lr[k], zs[(k + 0) * cols + o], s0);
                    s1 = fmaf(lr[k + 1], zs[(k + 1) * cols + o], s1);
                    s2 = fmaf(lr[k + 2], zs[(k + 2) * cols + o], s2);
                    s3 = fmaf(lr[k + 3], zs[(k + 3) * cols + o], s3);
                }
                for (; k < r; ++k) s0 = fmaf(lr[k], zs[k * cols + o], s0);
                zs[r * cols + o] = (cc[(size_t)(o0 + o) * in + r] - ((s0 + s1) + (s2 + s3))) / lr[r];
            }
            for (int r = in - 1; r >= 0; --r) {
                float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
                int k = r + 1;
                for (; k + 3 < in; k += 4) {
                    s0 = fmaf(Lp[at(k, r)], zs[k * cols + o], s0);
                    s1 = fmaf(Lp[at(k + 1, r)], zs[(k + 1) * cols + o], s1);
                    s2 = fmaf(Lp[at(k + 2, r)], zs[(k + 2) * cols + o], s2);
                    s3 = fmaf(Lp[at(k + 3, r)], zs[(k + 3) * cols + o], s3);
                }
                for (; k < in; ++k) s0 = fmaf(Lp[at(k, r)], zs[k * cols + o], s0);
                zs[r * cols + o] = (zs[r * cols + o] - ((s0 + s1) + (s2 + s3))) / Lp[at(r, r)];
            }
        }
        __syncthreads();
        for (int i = threadIdx.x; i < in * nc; i += blockDim.x) {
            const int r = i / nc, o = i - r * nc;
            w[off + (size_t)r * dt + o0 + o] = from_f32<T>(bad ? 0.f : zs[r * cols + o]);
        }
        __syncthreads();
    }
    if (bad && threadIdx.x == 0) set_status(status, kFitNotPosDef);
}

// solution columns per block for the small solve, and its dynamic shared memory
int small_solve_cols(int in, int dt)
{
    const int tri = in * (in + 1) / 2;
    const int cols = (kSmallSolveSmem / 4 - tri) / in;
    return cols < dt ? cols : dt;
}
size_t small_solve_smem(int in, int cols) { return ((size_t)in * (in + 1) / 2 + (size_t)in * cols) * sizeof(float); }

}  // namespace
}  // namespace kvx

using namespace kvx;

struct kvx_fitter {
    Geometry geo;
    int device = 0;
    int groups = 0, chunk = 0;
    double lambda = 0.0;
    long long tokens = 0;
    unsigned long long* rope = nullptr;   // device turns
    unsigned* status = nullptr;
    void* rows = nullptr;                 // X [groups][chunk][in] | Y [groups][chunk][dt]
    float* sums = nullptr;                // G [groups][in][in] | C [groups][dt][in]
    void* blas_ws = nullptr;
    cublasHandle_t blas = nullptr;
};

static const size_t kBlasWorkspace = 32u << 20;

static kvx_status fit_fail(kvx_status s, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
static kvx_status fit_fail(kvx_status s, const char* fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    set_last_error(buf);
    return s;
}

static void free_fitter(kvx_fitter* f)
{
    if (!f) return;
    if (f->blas) cublasDestroy(f->blas);
    if (f->blas_ws) cudaFree(f->blas_ws);
    if (f->rows) cudaFree(f->rows);
    if (f->sums) cudaFree(f->sums);
    if (f->rope) cudaFree(f->rope);
    if (f->status) cudaFree(f->status);
    delete f;
}

static size_t fit_elt(const kvx_fitter* f) { return f->geo.desc.dtype == KVX_BF16 ? 2 : 4; }
static size_t sums_floats(const kvx_fitter* f)
{
    const size_t in = f->geo.in_dim, dt = f->geo.desc.dst.head_dim;
    return (size_t)f->groups * in * (in + dt);
}

extern "C" KVX_API kvx_status kvx_fit_create(const kvx_translator_desc* desc, double lambda, int32_t chunk_tokens,
                                             kvx_fitter** out)
{
    if (!desc || !out) return fit_fail(KVX_ERR_INVALID_ARG, "fit_create: NULL argument");
    *out = nullptr;
    if (!(lambda >= 0.0)) return fit_fail(KVX_ERR_INVALID_ARG, "fit_create: lambda must be >= 0");
    if (chunk_tokens < 0 || chunk_tokens > (1 << 20))
        return fit_fail(KVX_ERR_INVALID_ARG, "fit_create: chunk_tokens outside [0, 1<<20]");
    char err[512];
    kvx_fitter* f = new kvx_fitter();
    kvx_status st = make_geometry(desc, "fit_create", f->geo, err);
    if (st != KVX_OK) {
        delete f;
        set_last_error(err);
        return st;
    }
    if (f->geo.in_dim > 512) {
        const int in_dim = f->geo.in_dim;
        delete f;
        return fit_fail(KVX_ERR_UNSUPPORTED, "fit_create: translator input width %d > 512", in_dim);
    }
    const kvx_translator_desc& D = f->geo.desc;
    f->lambda = lambda;
    f->chunk = chunk_tokens ? chunk_tokens : 4096;
    f->groups = D.dst.num_layers * D.dst.num_kv_heads * 2;
    const size_t in = f->geo.in_dim, dt = D.dst.head_dim;
    const size_t row_bytes = (size_t)f->groups * f->chunk * (in + dt) * fit_elt(f);
    const size_t rope_bytes = (size_t)(D.src.head_dim / 2 + D.dst.head_dim / 2) * sizeof(unsigned long long);
    cudaError_t ce;
    if (cudaGetDevice(&f->device) != cudaSuccess) { free_fitter(f); return fit_fail(KVX_ERR_CUDA, "fit_create: no CUDA device"); }
    if (cudaMalloc(&f->rows, row_bytes) != cudaSuccess || cudaMalloc(&f->sums, sums_floats(f) * sizeof(float)) != cudaSuccess ||
        cudaMalloc(&f->rope, rope_bytes) != cudaSuccess || cudaMalloc(&f->status, sizeof(unsigned)) != cudaSuccess ||
        cudaMalloc(&f->blas_ws, kBlasWorkspace) != cudaSuccess) {
        free_fitter(f);
        return fit_fail(KVX_ERR_OOM, "fit_create: device allocation (%zu bytes of rows)", row_bytes);
    }
    if ((ce = cudaMemcpy(f->rope, f->geo.turns, rope_bytes, cudaMemcpyHostToDevice)) != cudaSuccess ||
        (ce = cudaMemset(f->sums, 0, sums_floats(f) * sizeof(float))) != cudaSuccess ||
        (ce = cudaMemset(f->status, 0, sizeof(unsigned))) != cudaSuccess || (ce = cudaDeviceSynchronize()) != cudaSuccess) {
        free_fitter(f);
        return fit_fail(KVX_ERR_CUDA, "fit_create: %s", cudaGetErrorString(ce));
    }
    if (cublasCreate(&f->blas) != CUBLAS_STATUS_SUCCESS ||
        cublasSetWorkspace(f->blas, f->blas_ws, kBlasWorkspace) != CUBLAS_STATUS_SUCCESS) {
        free_fitter(f);
        return fit_fail(KVX_ERR_CUDA, "fit_create: cuBLAS initialisation");
    }
    *out = f;
    return KVX_OK;
}

extern "C" KVX_API kvx_status kvx_fit_accumulate(kvx_fitter* f, const kvx_src_kv* src, const kvx_tgt_tokens* tgt,
                                                 const kvx_dst_kv* target_cache, void* stream)
{
    if (!f || !src || !tgt || !target_cache) return fit_fail(KVX_ERR_INVALID_ARG, "fit_accumulate: NULL argument");
    TranslateParams P;
    char err[512];
    kvx_status st = make_params(f->geo, f->rope, f->status, nullptr, src, tgt, target_cache, P, "fit_accumulate", err);
    if (st != KVX_OK) {
        set_last_error(err);
        return st;
    }
    if (tgt->total_tokens == 0) return KVX_OK;
    const kvx_translator_desc& D = f->geo.desc;
    const int in = f->geo.in_dim, dt = D.dst.head_dim;
    const bool bf = D.dtype == KVX_BF16;
    const size_t elt = fit_elt(f);
    cudaStream_t s = (cudaStream_t)stream;
    if (cublasSetStream(f->blas, s) != CUBLAS_STATUS_SUCCESS)
        return fit_fail(KVX_ERR_CUDA, "fit_accumulate: cublasSetStream");
    char* xbase = (char*)f->rows;
    char* ybase = xbase + (size_t)f->groups * f->chunk * in * elt;
    float* G = f->sums;
    float* C = f->sums + (size_t)f->groups * in * in;
    const float one = 1.f;
    const cudaDataType_t ty = bf ? CUDA_R_16BF : CUDA_R_32F;
    for (int t0 = 0; t0 < tgt->total_tokens; t0 += f->chunk) {
        const int n = tgt->total_tokens - t0 < f->chunk ? tgt->total_tokens - t0 : f->chunk;
        FitRows R{xbase, ybase, f->chunk, t0, n};
        dim3 grid((n + kFitTile - 1) / kFitTile, D.dst.num_kv_heads, D.dst.num_layers * 2);
        if (bf) fit_rows_kernel<__nv_bfloat16><<<grid, kFitThreads, 0, s>>>(P, R);
        else fit_rows_kernel<float><<<grid, kFitThreads, 0, s>>>(P, R);
        cudaError_t ce = cudaGetLastError();
        if (ce != cudaSuccess) return fit_fail(KVX_ERR_CUDA, "fit_accumulate: %s", cudaGetErrorString(ce));
        // G[g] += X^T X: column-major X is in x n (ld in); C[g] += X^T Y with Y column-major dt x n (ld dt)
        cublasStatus_t bs = cublasGemmStridedBatchedEx(
            f->blas, CUBLAS_OP_N, CUBLAS_OP_T, in, in, n, &one, xbase, ty, in, (long long)f->chunk * in, xbase, ty, in,
            (long long)f->chunk * in, &one, G, CUDA_R_32F, in, (long long)in * in, f->groups, CUBLAS_COMPUTE_32F,
            CUBLAS_GEMM_DEFAULT);
        if (bs == CUBLAS_STATUS_SUCCESS)
            bs = cublasGemmStridedBatchedEx(f->blas, CUBLAS_OP_N, CUBLAS_OP_T, in, dt, n, &one, xbase, ty, in,
                                            (long long)f->chunk * in, ybase, ty, dt, (long long)f->chunk * dt, &one, C,
                                            CUDA_R_32F, in, (long long)in * dt, f->groups, CUBLAS_COMPUTE_32F,
                                            CUBLAS_GEMM_DEFAULT);
        if (bs != CUBLAS_STATUS_SUCCESS) return fit_fail(KVX_ERR_CUDA, "fit_accumulate: cuBLAS GEMM failed (%d)", (int)bs);
    }
    f->tokens += tgt->total_tokens;
    return KVX_OK;
}

extern "C" KVX_API kvx_status kvx_fit_solve(kvx_fitter* f, void* w_k, void* w_v, uint32_t* status_bits, void* stream)
{
    if (!f || !w_k || !w_v) return fit_fail(KVX_ERR_INVALID_ARG, "fit_solve: NULL argument");
    const kvx_translator_desc& D = f->geo.desc;
    const int in = f->geo.in_dim, dt = D.dst.head_dim;
    cudaStream_t s = (cudaStream_t)stream;
    // double scratch for the factorisation and the solutions: the row workspace is reused when it is
    // large enough, otherwise a temporary allocation (solve is not on the translation path)
    const size_t need = in <= kSmallSolve ? 0 : (size_t)f->groups * in * (in + dt) * sizeof(double);
    const size_t have = (size_t)f->groups * f->chunk * (in + dt) * fit_elt(f);
    double* scratch = nullptr;
    bool own = false;
    cudaError_t ce;
    if (need <= have) {
        scratch = (double*)f->rows;
    } else {
        if (cudaMalloc(&scratch, need) != cudaSuccess) return fit_fail(KVX_ERR_OOM, "fit_solve: scratch allocation");
        own = true;
    }
    double* A = scratch;
    double* Z = scratch + (size_t)f->groups * in * in;
    const float* G = f->sums;
    const float* C = f->sums + (size_t)f->groups * in * in;
    if (in <= kSmallSolve) {
        // fp32 factor and a block of solution columns in shared memory
        const int cols = small_solve_cols(in, dt);
        const int smem = (int)small_solve_smem(in, cols);
        if (D.dtype == KVX_BF16) {
            ce = cudaFuncSetAttribute(fit_solve_small_kernel<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
            if (ce == cudaSuccess)
                fit_solve_small_kernel<__nv_bfloat16><<<f->groups, kSmallSolveThreads, smem, s>>>(
                    G, C, (__nv_bfloat16*)w_k, (__nv_bfloat16*)w_v, in, dt, cols, (float)f->lambda, f->status);
        } else {
            ce = cudaFuncSetAttribute(fit_solve_small_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
            if (ce == cudaSuccess)
                fit_solve_small_kernel<float><<<f->groups, kSmallSolveThreads, smem, s>>>(
                    G, C, (float*)w_k, (float*)w_v, in, dt, cols, (float)f->lambda, f->status);
        }
        if (ce != cudaSuccess) {
            if (own) cudaFree(scratch);
            return fit_fail(KVX_ERR_CUDA, "fit_solve: %s", cudaGetErrorString(ce));
        }
    } else if (D.dtype == KVX_BF16)
        fit_solve_kernel<__nv_bfloat16><<<f->groups, kSolveThreads, 0, s>>>(G, C, A, Z, (__nv_bfloat16*)w_k,
                                                                            (__nv_bfloat16*)w_v, in, dt, f->lambda,
                                                                            f->status);
    else
        fit_solve_kernel<float><<<f->groups, kSolveThreads, 0, s>>>(G, C, A, Z, (float*)w_k, (float*)w_v, in, dt,
                                                                    f->lambda, f->status);
    unsigned bits = 0;
    if ((ce = cudaGetLastError()) != cudaSuccess || (ce = cudaStreamSynchronize(s)) != cudaSuccess ||
        (ce = cudaMemcpy(&bits, f->status, sizeof bits, cudaMemcpyDeviceToHost)) != cudaSuccess) {
        if (own) cudaFree(scratch);
        return fit_fail(KVX_ERR_CUDA, "fit_solve: %s", cudaGetErrorString(ce));
    }
    if (own) cudaFree(scratch);
    if (status_bits) *status_bits = bits;
    if (bits & kFitNotPosDef)
        return fit_fail(KVX_ERR_DEVICE_STATUS, "fit_solve: a system was not positive definite (status 0x%x)", bits);
    return KVX_OK;
}

extern "C" KVX_API kvx_status kvx_fit_reset(kvx_fitter* f, void* stream)
{
    if (!f) return fit_fail(KVX_ERR_INVALID_ARG, "fit_reset: NULL fitter");
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t ce;
    if ((ce = cudaMemsetAsync(f->sums, 0, sums_floats(f) * sizeof(float), s)) != cudaSuccess ||
        (ce = cudaMemsetAsync(f->status, 0, sizeof(unsigned), s)) != cudaSuccess)
        return fit_fail(KVX_ERR_CUDA, "fit_reset: %s", cudaGetErrorString(ce));
    f->tokens = 0;
    return KVX_OK;
}

extern "C" KVX_API int64_t kvx_fit_tokens(const kvx_fitter* f) { return f ? f->tokens : 0; }

extern "C" KVX_API kvx_status kvx_fit_destroy(kvx_fitter* f)
{
    if (!f) return KVX_OK;
    cudaDeviceSynchronize();
    free_fitter(f);
    return KVX_OK;
}
