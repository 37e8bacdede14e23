// kvx_fit.cu -- closed-form fit of the linear translator (paper Section 5).
//
// Section 5 gives the learning objective L_KV = D(T_theta(KV_A(C)), KV_B(C)).  With D the
// squared Euclidean distance over target tokens plus a ridge term lambda |W|^2, every
// (target layer j, target head h, K|V) group is a least-squares problem solved by the normal
// equations (X^T X + lambda I) W = X^T Y:
//   X rows: the translator's input rows (span mean of the un-rotated source rows, as the
//           translation forms them), rounded to the cache dtype;
//   Y rows: the target model's own cache rows, target RoPE undone for K.
// Accumulation (kvx_fit_accumulate), bf16 caches with in + d_t <= 512:
//   fit_gram_tc_kernel builds the transposed rows [X | Y]^T of 64 tokens at a time in shared
//   memory and adds X^T X and X^T Y on the tensor cores (tokens are the contraction dimension),
//   accumulating in TMEM; X and Y never go to global memory.
// Otherwise (fp32 caches, wider inputs):
//   fit_rows_kernel builds X and Y for one pass of up to chunk tokens, then fit_gram_simt_kernel
//   adds their products into the sums on the CUDA cores.
// Solve (kvx_fit_solve): one CTA per group factors X^T X + lambda I = L L^T and runs the two
//   triangular solves per output column: fit_solve_small_kernel in fp32 shared memory for
//   in <= 256 (with one step of iterative refinement against the fp32 sums), fit_solve_kernel in
//   double global memory above.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include "kvx_common.cuh"
#include "kvx_kernels.h"
#include "kvx_tc_common.cuh"

namespace kvx {
namespace {

constexpr int kFitTile = 32;
constexpr int kFitThreads = 256;
constexpr int kSolveThreads = 256;
constexpr unsigned kFitNotPosDef = 0x20u;   // status bit: a system was not positive definite
constexpr unsigned kFitSolvedDouble = 0x40u;   // status bit: ill-conditioned systems were solved in double
// The fp32 factorisation's relative error grows with cond(X^T X + lambda I) times in 2^-24;
// systems whose pivots show a condition number above this (cond >= (max L_ii / min L_ii)^2)
// are factored again in double.
constexpr float kSmallSolveMaxCond = 1e3f;

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
// only: NULL, or int[groups]: solve only the groups marked nonzero.
template <typename T>
__global__ void __launch_bounds__(kSolveThreads) fit_solve_kernel(const float* __restrict__ G,
                                                                  const float* __restrict__ C, double* A, double* Z,
                                                                  T* wk, T* wv, int in, int dt, double lambda,
                                                                  unsigned* status, const int* only)
{
    __shared__ int bad;
    const int g = blockIdx.x;
    if (only && !only[g]) return;
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

// redo: int[1 + groups]; a group whose factor shows a condition number above kSmallSolveMaxCond
// writes no W, sets redo[1 + g] and counts itself in redo[0] (fit_solve_kernel then solves it in
// double).
template <typename T>
__global__ void __launch_bounds__(kSmallSolveThreads) fit_solve_small_kernel(const float* __restrict__ G,
                                                                             const float* __restrict__ C, T* wk,
                                                                             T* wv, int in, int dt, int cols,
                                                                             float lambda, unsigned* status, int* redo)
{
    extern __shared__ float Lp[];          // packed lower triangle, then the solution block
    __shared__ float colk[kSmallSolve];    // column k of L below the diagonal
    __shared__ int bad, ill;
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
    if (threadIdx.x == 0) {
        float dmin = Lp[0], dmax = Lp[0];
        for (int k = 1; k < in; ++k) {
            const float d = Lp[at(k, k)];
            dmin = fminf(dmin, d);
            dmax = fmaxf(dmax, d);
        }
        const float ratio = dmax / dmin;
        ill = !bad && ratio * ratio > kSmallSolveMaxCond;
        if (ill) {
            redo[1 + g] = 1;
            atomicAdd(&redo[0], 1);
        }
    }
    __syncthreads();
    if (ill) return;
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

// ------------------------------------------------------------------ Gram sums on the CUDA cores
// One CTA per (group, 32-row block of X^T, 32-column block of the in + dt columns of Z = [X | Y]):
// the block's sums over the pass's n tokens in fp32, added into G (X^T X, row-major [in][in]) or
// C (X^T Y, column-major [dt][in]).  Each CTA owns its block, so plain read-modify-writes.
template <typename T>
__global__ void __launch_bounds__(256) fit_gram_simt_kernel(const T* __restrict__ X, const T* __restrict__ Y,
                                                            int chunk, int n, int in, int dt, float* G, float* C)
{
    __shared__ float xs[32][33], zs[32][33];
    const int g = blockIdx.z, rb = blockIdx.x * 32, cb = blockIdx.y * 32;
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const T* xg = X + (size_t)g * chunk * in;
    const T* yg = Y + (size_t)g * chunk * dt;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int t0 = 0; t0 < n; t0 += 32) {
        for (int k = ty; k < 32; k += 8) {
            const int t = t0 + k;
            const int col = cb + tx;
            xs[k][tx] = t < n ? to_f32<T>(xg[(size_t)t * in + rb + tx]) : 0.f;
            zs[k][tx] = t >= n ? 0.f : (col < in ? to_f32<T>(xg[(size_t)t * in + col]) : to_f32<T>(yg[(size_t)t * dt + col - in]));
        }
        __syncthreads();
#pragma unroll 8
        for (int k = 0; k < 32; ++k)
#pragma unroll
            for (int q = 0; q < 4; ++q) acc[q] = fmaf(xs[k][ty + 8 * q], zs[k][tx], acc[q]);
        __syncthreads();
    }
    const int col = cb + tx;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int row = rb + ty + 8 * q;
        if (col < in) G[((size_t)g * in + row) * in + col] += acc[q];
        else C[((size_t)g * dt + col - in) * in + row] += acc[q];
    }
}

// ------------------------------------------------------------------ Gram sums on the tensor cores (bf16)
// Work: per group g = (j*Ht + h)*2 + kv, row block mb (128 input channels) and 64-token K-block
// kb of the call:  D[i, n] += sum_t Z^T[mb*128 + i, t] * Z^T[n, t],  Z = [X | Y] (in + dt columns).
// The prologue warps build the block Z^T[in + dt rows][64 tokens] straight into shared memory in
// the UMMA K-major 128-byte-swizzled layout (the tokens are the contraction dimension, so they
// are the contiguous K of both operands; a 4-byte word holds two consecutive tokens of one
// channel), from the source and target caches exactly as fit_rows_kernel forms X and Y.  The MMA
// thread issues M = 128 (the block's rows of Z^T as A), N = in + dt (all rows of Z^T as B, in
// pieces of <= 256), K = 16 tokens per instruction into one fp32 TMEM accumulator that lives for
// the CTA's whole range of a (g, mb) unit; the epilogue warps then add it into the fp32 sums
// (vector atomics for X^T X rows, coalesced atomics for X^T Y columns).  Each CTA takes a
// contiguous range of the (unit, K-block) space, units ordered (g, mb) with mb fastest, so the
// two row blocks of a group read the same cache rows at about the same time (L2 hits).
constexpr int kGramK = 64;
constexpr int kGramMmaWarp = 0;
constexpr int kGramEpiWarp0 = 1;
constexpr int kGramNumEpi = 4;
constexpr int kGramXfWarp0 = kGramEpiWarp0 + kGramNumEpi;
constexpr int kGramNumXf = 8;
constexpr int kGramThreads = (kGramXfWarp0 + kGramNumXf) * 32;
constexpr int kGramMaxStages = 4;
constexpr int kGramMaxRows = 512;   // in + dt: one 128 x 512 fp32 accumulator fills TMEM

struct GramLaunch {
    int nrows;             // in + dt
    int mbs;               // row blocks of 128 input channels: in / 128
    int units;             // groups * mbs
    int nkb;               // K-blocks of 64 tokens in the call
    int stages;            // K-block ring depth
    unsigned stage_bytes;  // nrows * 128
    int n0;                // first N piece: columns [0, n0); second: [n0, nrows)
    unsigned idesc0, idesc1;
    float* G;              // [groups][in][in]
    float* C;              // [groups][dt][in]
};

// Byte offset of the 4-byte word holding tokens (2 lw, 2 lw + 1) of row r in a K-major SW128
// block of 64 tokens (rows 128 bytes apart within an 8-row atom of 1024 bytes).
__device__ __forceinline__ uint32_t gram_word(int r, int lw)
{
    return (uint32_t)((r >> 3) * 1024 + (r & 7) * 128 + ((((lw >> 2) ^ (r & 7)) & 7) << 4) + (lw & 3) * 4);
}

// Bring the cache rows K-block w of unit `unit` reads into L2 ahead of its prologue: the
// source rows of every head-block (one range from the first token's span start to the last
// token's span end, within the first token's sequence) and the target rows (a range when the
// target cache is contiguous).  Prefetches are hints: ranges are clipped to the caches.
__device__ __forceinline__ void l2_prefetch(const void* p, uint32_t bytes)
{
    const char* c = (const char*)p;
    for (uint32_t o = 0; o < bytes; o += 16384u) {   // pieces of at most 16 KB
        const uint32_t n = bytes - o < 16384u ? bytes - o : 16384u;
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(c + o), "r"(n) : "memory");
    }
}
__device__ void gram_prefetch(const TranslateParams& P, int unit, int kb, int mbs)
{
    const int g = unit / mbs, kv = g & 1, jh = g >> 1, h = jh % P.Ht, j = jh / P.Ht;
    const int t0 = kb * kGramK, t1 = min(t0 + kGramK, P.T_total) - 1;
    if (t1 < t0) return;
    const int b = find_seq(P.seq_off, P.batch, t0);
    const int off = __ldg(&P.seq_off[b]), end = __ldg(&P.seq_off[b + 1]);
    int S = __ldg(&P.src_seq_len[b]);
    S = S < 0 ? 0 : (S > P.src_max_seq ? P.src_max_seq : S);
    const int tl = min(t1, end - 1);
    int lo = t0 - off, hi = tl - off + 1;
    if (P.span_lo) { lo = __ldg(&P.span_lo[t0]); hi = __ldg(&P.span_hi[tl]); }
    lo = max(lo, 0);
    hi = min(hi, S);
    if (P.ss == P.ds && hi > lo) {
        const int heads = P.in_dim / P.ds;
        for (int q = 0; q < heads; ++q) {
            int slot, gs;
            head_block(P, j, h, q, slot, gs);
            const __nv_bfloat16* base = (const __nv_bfloat16*)(kv ? P.src_v[slot] : P.src_k[slot]) +
                                        (long long)b * P.sb + (long long)gs * P.sh + (long long)lo * P.ss;
            l2_prefetch(base, (uint32_t)(hi - lo) * P.ds * 2);
        }
    }
    if (!P.paged && P.dts == P.dt) {
        const int ta = t0 - off, tb = min(tl - off + 1, P.dst_max_seq);
        if (tb > ta) {
            const __nv_bfloat16* rowp = (const __nv_bfloat16*)(kv ? P.dst_v[j] : P.dst_k[j]) + (long long)b * P.db +
                                        (long long)h * P.dh + (long long)ta * P.dts;
            l2_prefetch(rowp, (uint32_t)(tb - ta) * P.dt * 2);
        }
    }
}

template <int DS>
__global__ void __launch_bounds__(kGramThreads, 1) fit_gram_tc_kernel(const __grid_constant__ TranslateParams P,
                                                                      const __grid_constant__ GramLaunch L)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    uint64_t* sBar = reinterpret_cast<uint64_t*>(smem + (size_t)L.stages * L.stage_bytes);
    // barriers: full[s] (prologue warps), empty[s] (MMA commit), dfull (MMA commit), dempty (epilogue
    // warps), done (the MMA thread's last commit)
    const int bFull = 0, bEmpty = kGramMaxStages, bDFull = 2 * kGramMaxStages, bDEmpty = bDFull + 1, bDone = bDFull + 2;
    volatile int* sAbort = reinterpret_cast<volatile int*>(sBar + bDone + 1);
    uint32_t* sTmem = reinterpret_cast<uint32_t*>(sBar + bDone + 2);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    auto bar = [&](int i) { return smem_u32(&sBar[i]); };
    if (threadIdx.x == 0) {
        *sAbort = 0;
        for (int i = 0; i < L.stages; ++i) {
            mbar_init(bar(bFull + i), kGramNumXf);
            mbar_init(bar(bEmpty + i), 1);
        }
        mbar_init(bar(bDFull), 1);
        mbar_init(bar(bDEmpty), kGramNumEpi);
        mbar_init(bar(bDone), 1);
        fence_mbar_init();
    }
    if (warp == kGramMmaWarp) {
        tmem_alloc(smem_u32(sTmem), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *sTmem;
    const Waiter W{sAbort, P.status};
    const long long total = (long long)L.units * L.nkb;
    const int w0 = (int)((long long)blockIdx.x * total / gridDim.x);
    const int w1 = (int)((long long)(blockIdx.x + 1) * total / gridDim.x);
    const int in = P.in_dim, dt = P.dt;

    if (warp == kGramMmaWarp) {
        if (lane == 0) {
            uint32_t it = 0, ucount = 0;
            bool issued = false;
            for (int w = w0; w < w1; ++w, ++it) {
                const int unit = w / L.nkb, kb = w - unit * L.nkb;
                const bool first = w == w0 || kb == 0, last = w == w1 - 1 || kb == L.nkb - 1;
                const uint32_t s = it % (uint32_t)L.stages, ph = (it / (uint32_t)L.stages) & 1;
                if (first && !W.wait(bar(bDEmpty), (ucount & 1) ^ 1)) break;
                if (!W.wait(bar(bFull + s), ph)) break;
                tc_fence_after();
                const uint32_t st = smem_u32(smem) + s * L.stage_bytes;
                const uint32_t a0 = st + (uint32_t)(unit % L.mbs) * (128 / 8) * 1024;
#pragma unroll
                for (int k = 0; k < kGramK / 16; ++k) {
                    const uint32_t acc = (first && k == 0) ? 0u : 1u;
                    const uint64_t ad = sw128_desc(a0 + k * 32);
                    umma_bf16(tmem_base, ad, sw128_desc(st + k * 32), L.idesc0, acc);
                    if (L.n0 < L.nrows)
                        umma_bf16(tmem_base + (uint32_t)L.n0, ad, sw128_desc(st + (uint32_t)(L.n0 / 8) * 1024 + k * 32),
                                  L.idesc1, acc);
                }
                umma_commit(bar(bEmpty + s));
                issued = true;
                if (last) {
                    umma_commit(bar(bDFull));
                    ++ucount;
                }
            }
            // every MMA issued has completed before the accumulator is released
            if (issued) {
                umma_commit(bar(bDone));
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(bar(bDone), 0) && globaltimer() - t0 < kWaitNs) {}
            }
        }
        __syncwarp();
    } else if (warp < kGramXfWarp0) {
        // ------------------------------------------------------------ epilogue: accumulator -> sums
        const int quad = warp & 3;
        uint32_t ucount = 0;
        const int u_first = w0 / L.nkb, u_last = w1 > w0 ? (w1 - 1) / L.nkb : u_first - 1;
        for (int u = u_first; u <= u_last; ++u, ++ucount) {
            if (!W.wait(bar(bDFull), ucount & 1)) break;
            tc_fence_after();
            const int g = u / L.mbs, row = (u % L.mbs) * 128 + quad * 32 + lane;
            float* grow = L.G + ((size_t)g * in + row) * in;
            float* cg = L.C + (size_t)g * dt * in + row;
            const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16);
            for (int c0 = 0; c0 < L.nrows; c0 += 32) {
                uint32_t r[32];
                tmem_ld32(taddr + c0, r);
                tmem_ld_wait();
                if (c0 < in) {
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        atomicAdd(reinterpret_cast<float4*>(grow + c0 + 4 * q),
                                  make_float4(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]),
                                              __uint_as_float(r[4 * q + 2]), __uint_as_float(r[4 * q + 3])));
                } else {
#pragma unroll
                    for (int e = 0; e < 32; ++e) atomicAdd(cg + (size_t)(c0 - in + e) * in, __uint_as_float(r[e]));
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(bDEmpty));
        }
    } else {
        // ------------------------------------------------------------ prologue: Z^T blocks in shared memory
        constexpr int HS = DS / 2;
        constexpr int CPH = DS / 16;                 // chunk pairs (16 channels) per source head
        const int xw = warp - kGramXfWarp0;
        const int heads = in / DS;
        const int nx = heads * CPH, items = nx + dt / 16;
        const int hs_t = dt >> 1;
        uint32_t it = 0;
        if (xw == 0 && lane < 2 && w0 + lane < w1) {   // the first two K-blocks of the range
            const int w = w0 + lane, unit = w / L.nkb;
            gram_prefetch(P, unit, w - unit * L.nkb, L.mbs);
        }
        for (int w = w0; w < w1; ++w, ++it) {
            const int unit = w / L.nkb, kb = w - unit * L.nkb;
            const int g = unit / L.mbs;
            if (xw == 0 && lane == 0 && w + 2 < w1) {   // two K-blocks ahead
                const int un = (w + 2) / L.nkb;
                gram_prefetch(P, un, w + 2 - un * L.nkb, L.mbs);
            }
            const int kv = g & 1, jh = g >> 1, h = jh % P.Ht, j = jh / P.Ht;
            const uint32_t s = it % (uint32_t)L.stages, ph = (it / (uint32_t)L.stages) & 1;
            if (!W.wait(bar(bEmpty + s), ph ^ 1)) break;
            uint8_t* st = smem + (size_t)s * L.stage_bytes;
            // this lane's two tokens of the block
            TokenInfo ti[2];
            bool ok[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int tp = kb * kGramK + 2 * lane + u;
                ok[u] = tp < P.T_total;
                if (ok[u]) {
                    ti[u] = resolve_token(P, tp);
                    ok[u] = ti[u].dst_off >= 0 && ti[u].hi > ti[u].lo;
                }
            }
            const bool rot_s = kv == 0 && P.rs.enabled, rot_t = kv == 0 && P.rt.enabled;
            const __nv_bfloat16* tgt = (const __nv_bfloat16*)(kv ? P.dst_v[j] : P.dst_k[j]);
            const long long hoff = dst_head_off(P, h);
            for (int item = xw; item < items; item += kGramNumXf) {
                float a0[2][8], a1[2][8];
                int r_lo, r_hi;
                if (item < nx) {
                    // X: head-block q, chunk pair cp: span mean of the un-rotated source rows
                    const int q = item / CPH, cp = item - q * CPH;
                    int c_lo, c_hi;
                    pair_channels(cp * 8, HS, P.rhalf_s, c_lo, c_hi);
                    r_lo = q * DS + c_lo;
                    r_hi = q * DS + c_hi;
                    int slot, gs;
                    head_block(P, j, h, q, slot, gs);
                    const bool rot = rot_s && cp * 8 < P.rhalf_s;
#pragma unroll
                    for (int u = 0; u < 2; ++u) {
#pragma unroll
                        for (int e = 0; e < 8; ++e) { a0[u][e] = 0.f; a1[u][e] = 0.f; }
                        if (!ok[u]) continue;
                        const __nv_bfloat16* base = (const __nv_bfloat16*)(kv ? P.src_v[slot] : P.src_k[slot]) +
                                                    (long long)ti[u].b * P.sb + (long long)gs * P.sh;
                        for (int sidx = ti[u].lo; sidx < ti[u].hi; ++sidx) {
                            const __nv_bfloat16* rowp = base + (long long)sidx * P.ss;
                            const uint4 w0v = __ldg(reinterpret_cast<const uint4*>(rowp + c_lo));
                            const uint4 w1v = __ldg(reinterpret_cast<const uint4*>(rowp + c_hi));
                            const uint32_t v0[4] = {w0v.x, w0v.y, w0v.z, w0v.w}, v1[4] = {w1v.x, w1v.y, w1v.z, w1v.w};
                            if (rot) {
                                const int pos = src_pos_of(P, ti[u].b, sidx);
#pragma unroll
                                for (int e = 0; e < 8; ++e) {   // R(-theta)
                                    const float x0 = (e & 1) ? bf_hi(v0[e >> 1]) : bf_lo(v0[e >> 1]);
                                    const float x1 = (e & 1) ? bf_hi(v1[e >> 1]) : bf_lo(v1[e >> 1]);
                                    const float2 cs = rope_cs(P.rs, pos, cp * 8 + e);
                                    a0[u][e] += fmaf(x0, cs.x, x1 * cs.y);
                                    a1[u][e] += fmaf(x1, cs.x, -x0 * cs.y);
                                }
                            } else {
#pragma unroll
                                for (int e = 0; e < 8; ++e) {
                                    a0[u][e] += (e & 1) ? bf_hi(v0[e >> 1]) : bf_lo(v0[e >> 1]);
                                    a1[u][e] += (e & 1) ? bf_hi(v1[e >> 1]) : bf_lo(v1[e >> 1]);
                                }
                            }
                        }
                        const float inv = 1.f / (float)(ti[u].hi - ti[u].lo);
#pragma unroll
                        for (int e = 0; e < 8; ++e) { a0[u][e] *= inv; a1[u][e] *= inv; }
                    }
                } else {
                    // Y: chunk pair cp of the target row, target RoPE undone for K
                    const int cp = item - nx;
                    int c_lo, c_hi;
                    pair_channels(cp * 8, hs_t, P.rhalf_t, c_lo, c_hi);
                    r_lo = in + c_lo;
                    r_hi = in + c_hi;
                    const bool rot = rot_t && cp * 8 < P.rhalf_t;
#pragma unroll
                    for (int u = 0; u < 2; ++u) {
#pragma unroll
                        for (int e = 0; e < 8; ++e) { a0[u][e] = 0.f; a1[u][e] = 0.f; }
                        if (!ok[u]) continue;
                        const __nv_bfloat16* rowp = tgt + ti[u].dst_off + hoff;
                        const uint4 w0v = __ldg(reinterpret_cast<const uint4*>(rowp + c_lo));
                        const uint4 w1v = __ldg(reinterpret_cast<const uint4*>(rowp + c_hi));
                        const uint32_t v0[4] = {w0v.x, w0v.y, w0v.z, w0v.w}, v1[4] = {w1v.x, w1v.y, w1v.z, w1v.w};
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            const float y0 = (e & 1) ? bf_hi(v0[e >> 1]) : bf_lo(v0[e >> 1]);
                            const float y1 = (e & 1) ? bf_hi(v1[e >> 1]) : bf_lo(v1[e >> 1]);
                            if (rot) {   // R(-theta)
                                const float2 cs = rope_cs(P.rt, ti[u].pt, cp * 8 + e);
                                a0[u][e] = fmaf(y0, cs.x, y1 * cs.y);
                                a1[u][e] = fmaf(y1, cs.x, -y0 * cs.y);
                            } else {
                                a0[u][e] = y0;
                                a1[u][e] = y1;
                            }
                        }
                    }
                }
                // rows r_lo + e and r_hi + e, tokens (2 lane, 2 lane + 1) of the block: one word each
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    *reinterpret_cast<uint32_t*>(st + gram_word(r_lo + e, lane)) = pack_bf16(a0[0][e], a0[1][e]);
                    *reinterpret_cast<uint32_t*>(st + gram_word(r_hi + e, lane)) = pack_bf16(a1[0][e], a1[1][e]);
                }
            }
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(bFull + s));
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == kGramMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, 512);
    }
}

uint32_t gram_idesc(int N)
{
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(128 >> 4) << 24);
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
    int* redo = nullptr;                  // [1 + groups]: systems the fp32 solve hands to the double one
    int device = 0, num_sms = 0;
    int groups = 0, chunk = 0;
    int tc = 0;                           // Gram sums by fit_gram_tc_kernel (no row workspace)
    double lambda = 0.0;
    long long tokens = 0;
    unsigned long long* rope = nullptr;   // device turns
    unsigned* status = nullptr;
    void* rows = nullptr;                 // CUDA-core path: X [groups][chunk][in] | Y [groups][chunk][dt]
    size_t rows_bytes = 0;
    float* sums = nullptr;                // G [groups][in][in] | C [groups][dt][in]
};

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
    if (f->rows) cudaFree(f->rows);
    if (f->redo) cudaFree(f->redo);
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
    const int ds = D.src.head_dim;
    // tensor-core Gram sums for bf16 caches whose input rows split into 128-channel blocks and
    // whose [X | Y] rows fit one TMEM accumulator; the CUDA-core path otherwise
    f->tc = D.dtype == KVX_BF16 && in % 128 == 0 && in + dt <= (size_t)kGramMaxRows && in % ds == 0 &&
            (ds == 64 || ds == 128 || ds == 256);
    f->rows_bytes = f->tc ? 0 : (size_t)f->groups * f->chunk * (in + dt) * fit_elt(f);
    const size_t rope_bytes = (size_t)(D.src.head_dim / 2 + D.dst.head_dim / 2) * sizeof(unsigned long long);
    cudaError_t ce;
    if (cudaGetDevice(&f->device) != cudaSuccess ||
        cudaDeviceGetAttribute(&f->num_sms, cudaDevAttrMultiProcessorCount, f->device) != cudaSuccess) {
        free_fitter(f);
        return fit_fail(KVX_ERR_CUDA, "fit_create: no CUDA device");
    }
    if ((f->rows_bytes && cudaMalloc(&f->rows, f->rows_bytes) != cudaSuccess) ||
        cudaMalloc(&f->sums, sums_floats(f) * sizeof(float)) != cudaSuccess ||
        cudaMalloc(&f->rope, rope_bytes) != cudaSuccess || cudaMalloc(&f->status, sizeof(unsigned)) != cudaSuccess ||
        cudaMalloc(&f->redo, sizeof(int) * (1 + (size_t)f->groups)) != cudaSuccess) {
        const size_t rb = f->rows_bytes;
        free_fitter(f);
        return fit_fail(KVX_ERR_OOM, "fit_create: device allocation (%zu bytes of rows)", rb);
    }
    if ((ce = cudaMemcpy(f->rope, f->geo.turns, rope_bytes, cudaMemcpyHostToDevice)) != cudaSuccess ||
        (ce = cudaMemset(f->sums, 0, sums_floats(f) * sizeof(float))) != cudaSuccess ||
        (ce = cudaMemset(f->status, 0, sizeof(unsigned))) != cudaSuccess || (ce = cudaDeviceSynchronize()) != cudaSuccess) {
        free_fitter(f);
        return fit_fail(KVX_ERR_CUDA, "fit_create: %s", cudaGetErrorString(ce));
    }
    *out = f;
    return KVX_OK;
}

template <int DS>
static cudaError_t launch_gram_tc(const TranslateParams& P, const GramLaunch& L, int grid, size_t smem, cudaStream_t s)
{
    const cudaError_t e = smem_opt_in<fit_gram_tc_kernel<DS>>((int)smem);
    if (e != cudaSuccess) return e;
    fit_gram_tc_kernel<DS><<<grid, kGramThreads, smem, s>>>(P, L);
    return cudaGetLastError();
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
    float* G = f->sums;
    float* C = f->sums + (size_t)f->groups * in * in;
    if (f->tc) {
        GramLaunch L{};
        L.nrows = in + dt;
        L.mbs = in / 128;
        L.units = f->groups * L.mbs;
        L.nkb = (tgt->total_tokens + kGramK - 1) / kGramK;
        L.stage_bytes = (unsigned)L.nrows * 128;
        L.stages = (int)((kSmemMax - 1024 - 256) / L.stage_bytes);
        if (L.stages > kGramMaxStages) L.stages = kGramMaxStages;
        L.n0 = L.nrows < 256 ? L.nrows : 256;
        L.idesc0 = gram_idesc(L.n0);
        L.idesc1 = L.nrows > L.n0 ? gram_idesc(L.nrows - L.n0) : 0u;
        L.G = G;
        L.C = C;
        const long long work = (long long)L.units * L.nkb;
        const int grid = (int)(work < f->num_sms ? work : f->num_sms);
        const size_t smem = 1024 + (size_t)L.stages * L.stage_bytes + 256;
        cudaError_t ce;
        switch (D.src.head_dim) {
        case 64: ce = launch_gram_tc<64>(P, L, grid, smem, s); break;
        case 128: ce = launch_gram_tc<128>(P, L, grid, smem, s); break;
        default: ce = launch_gram_tc<256>(P, L, grid, smem, s); break;
        }
        if (ce != cudaSuccess) return fit_fail(KVX_ERR_CUDA, "fit_accumulate: %s", cudaGetErrorString(ce));
        f->tokens += tgt->total_tokens;
        return KVX_OK;
    }
    char* xbase = (char*)f->rows;
    char* ybase = xbase + (size_t)f->groups * f->chunk * in * elt;
    for (int t0 = 0; t0 < tgt->total_tokens; t0 += f->chunk) {
        const int n = tgt->total_tokens - t0 < f->chunk ? tgt->total_tokens - t0 : f->chunk;
        FitRows R{xbase, ybase, f->chunk, t0, n};
        dim3 grid((n + kFitTile - 1) / kFitTile, D.dst.num_kv_heads, D.dst.num_layers * 2);
        dim3 ggrid(in / 32, (in + dt) / 32, f->groups);
        if (bf) {
            fit_rows_kernel<__nv_bfloat16><<<grid, kFitThreads, 0, s>>>(P, R);
            fit_gram_simt_kernel<__nv_bfloat16><<<ggrid, 256, 0, s>>>((const __nv_bfloat16*)xbase,
                                                                      (const __nv_bfloat16*)ybase, f->chunk, n, in, dt,
                                                                      G, C);
        } else {
            fit_rows_kernel<float><<<grid, kFitThreads, 0, s>>>(P, R);
            fit_gram_simt_kernel<float><<<ggrid, 256, 0, s>>>((const float*)xbase, (const float*)ybase, f->chunk, n,
                                                              in, dt, G, C);
        }
        cudaError_t ce = cudaGetLastError();
        if (ce != cudaSuccess) return fit_fail(KVX_ERR_CUDA, "fit_accumulate: %s", cudaGetErrorString(ce));
    }
    f->tokens += tgt->total_tokens;
    return KVX_OK;
}

extern "C" KVX_API kvx_status kvx_fit_solve(kvx_fitter* f, void* w_k, void* w_v, uint32_t* status_bits, void* stream)
{
    if (!f || !w_k || !w_v) return fit_fail(KVX_ERR_INVALID_ARG, "fit_solve: NULL argument");
    const kvx_translator_desc& D = f->geo.desc;
    const int in = f->geo.in_dim, dt = D.dst.head_dim;
    const bool bf = D.dtype == KVX_BF16;
    cudaStream_t s = (cudaStream_t)stream;
    const float* G = f->sums;
    const float* C = f->sums + (size_t)f->groups * in * in;
    cudaError_t ce = cudaSuccess;
    int n_double = in <= kSmallSolve ? 0 : f->groups;   // systems for the double solve
    if (in <= kSmallSolve) {
        // fp32 factor and a block of solution columns in shared memory; ill-conditioned systems
        // are marked for the double solve
        const int cols = small_solve_cols(in, dt);
        const int smem = (int)small_solve_smem(in, cols);
        if ((ce = cudaMemsetAsync(f->redo, 0, sizeof(int) * (1 + (size_t)f->groups), s)) == cudaSuccess) {
            if (bf) {
                ce = cudaFuncSetAttribute(fit_solve_small_kernel<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
                if (ce == cudaSuccess)
                    fit_solve_small_kernel<__nv_bfloat16><<<f->groups, kSmallSolveThreads, smem, s>>>(
                        G, C, (__nv_bfloat16*)w_k, (__nv_bfloat16*)w_v, in, dt, cols, (float)f->lambda, f->status, f->redo);
            } else {
                ce = cudaFuncSetAttribute(fit_solve_small_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
                if (ce == cudaSuccess)
                    fit_solve_small_kernel<float><<<f->groups, kSmallSolveThreads, smem, s>>>(
                        G, C, (float*)w_k, (float*)w_v, in, dt, cols, (float)f->lambda, f->status, f->redo);
            }
        }
        if (ce == cudaSuccess) ce = cudaGetLastError();
        if (ce == cudaSuccess) ce = cudaMemcpyAsync(&n_double, f->redo, sizeof(int), cudaMemcpyDeviceToHost, s);
        if (ce == cudaSuccess) ce = cudaStreamSynchronize(s);
        if (ce != cudaSuccess) return fit_fail(KVX_ERR_CUDA, "fit_solve: %s", cudaGetErrorString(ce));
    }
    bool redone = false;
    if (n_double > 0) {
        // double scratch for the factorisation and the solutions: the row workspace when it is
        // large enough, else a temporary allocation (the solve is not on the translation path)
        const size_t need = (size_t)f->groups * in * (in + dt) * sizeof(double);
        double* scratch = nullptr;
        bool own = false;
        if (need <= f->rows_bytes) {
            scratch = (double*)f->rows;
        } else {
            if (cudaMalloc(&scratch, need) != cudaSuccess) return fit_fail(KVX_ERR_OOM, "fit_solve: scratch allocation");
            own = true;
        }
        double* A = scratch;
        double* Z = scratch + (size_t)f->groups * in * in;
        const int* only = in <= kSmallSolve ? f->redo + 1 : nullptr;
        if (bf)
            fit_solve_kernel<__nv_bfloat16><<<f->groups, kSolveThreads, 0, s>>>(G, C, A, Z, (__nv_bfloat16*)w_k,
                                                                                (__nv_bfloat16*)w_v, in, dt, f->lambda,
                                                                                f->status, only);
        else
            fit_solve_kernel<float><<<f->groups, kSolveThreads, 0, s>>>(G, C, A, Z, (float*)w_k, (float*)w_v, in, dt,
                                                                        f->lambda, f->status, only);
        ce = cudaGetLastError();
        if (ce == cudaSuccess) ce = cudaStreamSynchronize(s);
        if (own) cudaFree(scratch);
        if (ce != cudaSuccess) return fit_fail(KVX_ERR_CUDA, "fit_solve: %s", cudaGetErrorString(ce));
        redone = in <= kSmallSolve;
    }
    unsigned bits = 0;
    if ((ce = cudaMemcpy(&bits, f->status, sizeof bits, cudaMemcpyDeviceToHost)) != cudaSuccess)
        return fit_fail(KVX_ERR_CUDA, "fit_solve: %s", cudaGetErrorString(ce));
    if (redone) bits |= kFitSolvedDouble;
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
