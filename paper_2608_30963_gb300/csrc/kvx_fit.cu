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
//   fit_gram_tc_kernel builds the rows [X | Y] of 64 tokens at a time in shared memory and adds
//   X^T X and X^T Y on the tensor cores (tokens are the contraction dimension), accumulating in
//   TMEM; X and Y never go to global memory.
// Otherwise (fp32 caches, wider inputs):
//   fit_rows_kernel builds X and Y for one pass of up to chunk tokens, then fit_gram_simt_kernel
//   adds their products into the sums on the CUDA cores.
// Solve (kvx_fit_solve): one CTA per group factors X^T X + lambda I = L L^T and runs the two
//   triangular solves per output column: fit_solve_small_kernel in fp32 shared memory for
//   in <= 256, handing the systems whose factor shows a condition number above 10^3 to
//   fit_solve_kernel, which solves in double in global memory (and solves every system above
//   in = 256).
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
// kb of the call:  D[i, n] += sum_t Z^T[mb*128 + i, t] * Z^T[n, t],  Z = [X | Y].  Only the
// lower triangle of X^T X is formed (the solves read it): row block mb takes the X columns
// [0, (mb+1)*128) and the dt columns of Y, so its accumulator holds (mb+1)*128 + dt columns.
//   loader warp  resolves the block's 64 tokens into a table in shared memory.  For a call with
//                spans it also copies the block's source window (one bulk copy per source head
//                when the rows are contiguous) and its 64 target rows (one bulk copy when they are
//                consecutive) into a ring of raw slots.
//   12 prologue warps  build the block [X | Y] of 64 token rows, channels contiguous, in
//                128-byte-swizzled atoms of 64 channels x 8 tokens: the layout tcgen05 reads as
//                an MN-major operand, so both A and B are this block and nothing is transposed.
//                X rows as the translation forms them (span mean of un-rotated source rows), Y
//                rows with the target RoPE undone for K, both rounded to bf16.
//                With spans: all 12 warps on one block, lanes across a row's 16-channel chunk
//                pairs (8 lanes per 128-channel head), each lane taking the span mean of its
//                chunk pair; tokens whose span leaves the window read their rows from global
//                memory.
//                Identity alignment ("direct" blocks): 4 teams of 3 warps, one block per team.
//                A thread gathers its (token, chunk pair) items straight into their swizzled
//                places with 16-byte cp.async, waits for its own copies and un-rotates K in
//                place, one (cos, sin) per pair for every source head and, when the rotations
//                and the token's positions coincide, for its target row too.
//   MMA thread   M = 128 (the row block's channels as A), N over the needed columns (B, in
//                pieces of <= 256), K = 16 tokens per instruction, into one fp32 TMEM
//                accumulator that lives for the CTA's range of a unit.
//   4 epilogue warps  add the accumulator into the fp32 sums (vector atomics for X^T X rows,
//                coalesced atomics for X^T Y columns).
// Units are (g, chunk of K-blocks, mb) with mb fastest; each CTA takes an equal contiguous
// range of the (unit, K-block) space, so a range may start or end inside a unit.
constexpr int kGramK = 64;
constexpr int kGramMmaWarp = 0;
constexpr int kGramEpiWarp0 = 1;
constexpr int kGramNumEpi = 4;
constexpr int kGramXfWarp0 = kGramEpiWarp0 + kGramNumEpi;
// prologue warps: 12 for staged blocks, 16 (4 teams of 4) for direct blocks, whose prologue needs
// fewer registers (the CTA's 22 warps leave 88 a thread)
__host__ __device__ constexpr int gram_num_xf(bool direct) { return direct ? 16 : 12; }
__host__ __device__ constexpr int gram_load_warp(bool direct) { return kGramXfWarp0 + gram_num_xf(direct); }
__host__ __device__ constexpr int gram_threads(bool direct) { return (gram_load_warp(direct) + 1) * 32; }
constexpr int kGramMaxStages = 4;
constexpr int kGramMaxRaw = 8;
// Direct blocks (every span one source row): the prologue warps work in teams, one 64-token block each.
constexpr int kGramTeams = 4;
constexpr int kGramMaxRows = 512;   // in + dt: one 128 x 512 fp32 accumulator fills TMEM
constexpr int kGramMaxHeads = 6;    // source head-blocks in one input row

struct GramTok {
    int b, lo, hi, pt;       // sequence, clamped source span, target position
    long long dst_off;       // target row offset (head 0), -1: none
    int ok;                  // contributes (a valid row with a span)
    int ps;                  // direct blocks: source position of the span's row
};

struct GramLaunch {
    int nrows;             // in + dt (rows of a full Z^T block)
    int mbs;               // row blocks of 128 input channels: in / 128
    int nkb;               // K-blocks of 64 tokens in the call
    int kc;                // K-blocks per unit (a chunk); nkb % kc == 0
    int nch;               // chunks: nkb / kc
    int units;             // groups * nch * mbs
    int stages;            // Z^T block ring depth
    unsigned stage_bytes;  // nrows * 128
    int raw_slots;         // raw staging ring depth
    int rcap;              // source rows one window holds
    unsigned src_row, tgt_row;   // padded row pitches of the staged source / target rows (bytes)
    unsigned raw_bytes;    // one raw slot: token table, header, source window, target rows
    unsigned off_raw, off_bar;
    unsigned lbo, sbo;     // MN-major operand strides: between 64-channel blocks, between 8-token groups
    float* G;              // [groups][in][in]
    float* C;              // [groups][dt][in]
};

// Instruction descriptor: bf16 A and B, fp32 D, M = 128, N; both operands MN-major (bits 15, 16):
// the block holds token rows with the channels contiguous, and the contraction runs over tokens.
__host__ __device__ inline uint32_t gram_idesc_dev(int N)
{
    return (1u << 4) | (1u << 7) | (1u << 10) | (1u << 15) | (1u << 16) | ((uint32_t)(N >> 3) << 17) |
           ((uint32_t)(128 >> 4) << 24);
}
// Shared-memory descriptor of an MN-major operand in 128-byte-swizzled atoms of 64 channels x 8
// tokens: lbo between consecutive 64-channel blocks, sbo between consecutive 8-token groups.
__device__ __forceinline__ uint64_t sw128_mn_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// Byte offset of the 16-byte chunk of channels [c, c + 8) (c a multiple of 8) of token i in a block:
// 64-channel column blocks of 64 tokens x 128 bytes, 128-byte-swizzled in atoms of 8 tokens.
__device__ __forceinline__ uint32_t gram_chunk(int i, int c)
{
    return (uint32_t)((c >> 6) * (kGramK * 128) + (i >> 3) * 1024 + (i & 7) * 128 + ((((c >> 3) & 7) ^ (i & 7)) << 4));
}

// Unit u of the (g, chunk, mb) space and K-block index within the unit.
struct GramUnit {
    int g, mb, kb;   // kb: K-block of the call
};
__device__ __forceinline__ GramUnit gram_unit(const GramLaunch& L, int w)
{
    const int u = w / L.kc, kbi = w - u * L.kc;
    const int mb = u % L.mbs, gc = u / L.mbs;
    const int ch = gc % L.nch, g = gc / L.nch;
    return GramUnit{g, mb, ch * L.kc + kbi};
}

// Channels [c_lo, +8) and [c_hi, +8) of token i, rounded to bf16, into the block.
__device__ __forceinline__ void gram_put(uint8_t* st, int i, int c_lo, int c_hi, const float (&lo)[8], const float (&hi)[8])
{
    *reinterpret_cast<uint4*>(st + gram_chunk(i, c_lo)) =
        make_uint4(pack_bf16(lo[0], lo[1]), pack_bf16(lo[2], lo[3]), pack_bf16(lo[4], lo[5]), pack_bf16(lo[6], lo[7]));
    *reinterpret_cast<uint4*>(st + gram_chunk(i, c_hi)) =
        make_uint4(pack_bf16(hi[0], hi[1]), pack_bf16(hi[2], hi[3]), pack_bf16(hi[4], hi[5]), pack_bf16(hi[6], hi[7]));
}

// Rotates the 8 channel pairs of the chunks at lo and hi of a block in place by R(-theta).
__device__ __forceinline__ void gram_unrotate(uint8_t* lo, uint8_t* hi, const float2 (&cs)[8])
{
    const uint4 a = *reinterpret_cast<const uint4*>(lo), b = *reinterpret_cast<const uint4*>(hi);
    const uint32_t va[4] = {a.x, a.y, a.z, a.w}, vb[4] = {b.x, b.y, b.z, b.w};
    float y0[8], y1[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const float u0 = (e & 1) ? bf_hi(va[e >> 1]) : bf_lo(va[e >> 1]);
        const float u1 = (e & 1) ? bf_hi(vb[e >> 1]) : bf_lo(vb[e >> 1]);
        y0[e] = fmaf(u0, cs[e].x, u1 * cs[e].y);
        y1[e] = fmaf(u1, cs[e].x, -u0 * cs[e].y);
    }
    *reinterpret_cast<uint4*>(lo) =
        make_uint4(pack_bf16(y0[0], y0[1]), pack_bf16(y0[2], y0[3]), pack_bf16(y0[4], y0[5]), pack_bf16(y0[6], y0[7]));
    *reinterpret_cast<uint4*>(hi) =
        make_uint4(pack_bf16(y1[0], y1[1]), pack_bf16(y1[2], y1[3]), pack_bf16(y1[4], y1[5]), pack_bf16(y1[6], y1[7]));
}

// DS: source head dim; NHD: source head-blocks in one input row (in / DS).  DIRECT: identity
// alignment (every span one source row): the loader writes token tables only, and the prologue
// teams gather the rows with 16-byte asynchronous copies straight into the block.
template <int DS, int NHD, bool DIRECT>
__global__ void __launch_bounds__(gram_threads(DIRECT), 1) fit_gram_tc_kernel(const __grid_constant__ TranslateParams P,
                                                                      const __grid_constant__ GramLaunch L)
{
    constexpr int kGramNumXf = gram_num_xf(DIRECT);
    constexpr int kGramLoadWarp = gram_load_warp(DIRECT);
    constexpr int kGramTeamWarps = kGramNumXf / kGramTeams;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    uint8_t* sRaw = smem + L.off_raw;
    uint64_t* sBar = reinterpret_cast<uint64_t*>(smem + L.off_bar);
    // barriers: zfull[s] (prologue warps), zempty[s] (MMA commit), rfull[r] (loader + copies),
    // rempty[r] (prologue warps), dfull (MMA commit), dempty (epilogue warps), done (MMA)
    constexpr int bZFull = 0, bZEmpty = kGramMaxStages, bRFull = 2 * kGramMaxStages, bREmpty = bRFull + kGramMaxRaw;
    constexpr int bDFull = bREmpty + kGramMaxRaw, bDEmpty = bDFull + 1, bDone = bDFull + 2;
    volatile int* sAbort = reinterpret_cast<volatile int*>(sBar + bDone + 1);
    uint32_t* sTmem = reinterpret_cast<uint32_t*>(sBar + bDone + 2);
    unsigned long long* sTurn = reinterpret_cast<unsigned long long*>(sBar + bDone + 4);   // source | target
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    auto bar = [&](int i) { return smem_u32(&sBar[i]); };
    if (threadIdx.x == 0) {
        *sAbort = 0;
        for (int i = 0; i < L.stages; ++i) {
            mbar_init(bar(bZFull + i), DIRECT ? kGramTeamWarps : kGramNumXf);
            mbar_init(bar(bZEmpty + i), 1);
        }
        for (int i = 0; i < L.raw_slots; ++i) {
            mbar_init(bar(bRFull + i), 1);
            mbar_init(bar(bREmpty + i), DIRECT ? kGramTeamWarps : kGramNumXf);
        }
        mbar_init(bar(bDFull), 1);
        mbar_init(bar(bDEmpty), kGramNumEpi);
        mbar_init(bar(bDone), 1);
        fence_mbar_init();
    }
    for (int i = threadIdx.x; i < (P.ds >> 1); i += blockDim.x) sTurn[i] = P.rs.enabled ? __ldg(&P.rs.turns[i]) : 0ull;
    for (int i = threadIdx.x; i < (P.dt >> 1); i += blockDim.x)
        sTurn[(P.ds >> 1) + i] = P.rt.enabled ? __ldg(&P.rt.turns[i]) : 0ull;
    if (warp == kGramMmaWarp) {
        tmem_alloc(smem_u32(sTmem), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *sTmem;
    const Waiter W{sAbort, P.status};
    const long long total = (long long)L.units * L.kc;
    const int w0 = (int)((long long)blockIdx.x * total / gridDim.x);
    const int w1 = (int)((long long)(blockIdx.x + 1) * total / gridDim.x);
    const int in = NHD * DS, dt = P.dt;
    constexpr int heads = NHD;
    auto tok_tab = [&](int r) { return reinterpret_cast<GramTok*>(sRaw + (size_t)r * L.raw_bytes); };
    auto win_hdr = [&](int r) { return reinterpret_cast<int*>(sRaw + (size_t)r * L.raw_bytes + kGramK * sizeof(GramTok)); };
    auto src_rows = [&](int r, int q) {
        return sRaw + (size_t)r * L.raw_bytes + kGramK * sizeof(GramTok) + 16 + (size_t)q * L.rcap * L.src_row;
    };
    auto tgt_rows = [&](int r) {
        return sRaw + (size_t)r * L.raw_bytes + kGramK * sizeof(GramTok) + 16 + (size_t)heads * L.rcap * L.src_row;
    };

    if (warp == kGramMmaWarp) {
        if (lane == 0) {
            uint32_t it = 0, ucount = 0;
            bool issued = false;
            for (int w = w0; w < w1; ++w, ++it) {
                const GramUnit x = gram_unit(L, w);
                const int kbi = w % L.kc;
                const bool first = w == w0 || kbi == 0, last = w == w1 - 1 || kbi == L.kc - 1;
                const uint32_t s = it % (uint32_t)L.stages, ph = (it / (uint32_t)L.stages) & 1;
                if (first && !W.wait(bar(bDEmpty), (ucount & 1) ^ 1)) break;
                if (!W.wait(bar(bZFull + s), ph)) break;
                tc_fence_after();
                const uint32_t st = smem_u32(smem) + s * L.stage_bytes;
                const uint32_t colblk = kGramK * 128;            // one 64-channel column block
                const uint32_t a0 = st + (uint32_t)(x.mb * 2) * colblk;
                const int nx = (x.mb + 1) * 128;   // X columns of the lower triangle
#pragma unroll
                for (int k = 0; k < kGramK / 16; ++k) {   // 16 tokens = two 8-token atom rows
                    const uint32_t acc = (first && k == 0) ? 0u : 1u;
                    const uint64_t ad = sw128_mn_desc(a0 + k * 2048, L.lbo, L.sbo);
                    for (int c0 = 0; c0 < nx; c0 += 256) {   // X columns in pieces of <= 256
                        const int n = nx - c0 < 256 ? nx - c0 : 256;
                        umma_bf16(tmem_base + (uint32_t)c0, ad,
                                  sw128_mn_desc(st + (uint32_t)(c0 / 64) * colblk + k * 2048, L.lbo, L.sbo),
                                  gram_idesc_dev(n), acc);
                    }
                    umma_bf16(tmem_base + (uint32_t)nx, ad,
                              sw128_mn_desc(st + (uint32_t)(in / 64) * colblk + k * 2048, L.lbo, L.sbo),
                              gram_idesc_dev(dt), acc);
                }
                umma_commit(bar(bZEmpty + s));
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
        const int u_first = w0 / L.kc, u_last = w1 > w0 ? (w1 - 1) / L.kc : u_first - 1;
        for (int u = u_first; u <= u_last; ++u, ++ucount) {
            if (!W.wait(bar(bDFull), ucount & 1)) break;
            tc_fence_after();
            const GramUnit x = gram_unit(L, u * L.kc);
            const int nx = (x.mb + 1) * 128;
            const int row = x.mb * 128 + quad * 32 + lane;
            float* grow = L.G + ((size_t)x.g * in + row) * in;
            float* cg = L.C + (size_t)x.g * dt * in + row;
            const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16);
            for (int c0 = 0; c0 < nx + dt; c0 += 32) {
                uint32_t r[32];
                tmem_ld32(taddr + c0, r);
                tmem_ld_wait();
                if (c0 < nx) {
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        atomicAdd(reinterpret_cast<float4*>(grow + c0 + 4 * q),
                                  make_float4(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]),
                                              __uint_as_float(r[4 * q + 2]), __uint_as_float(r[4 * q + 3])));
                } else {
#pragma unroll
                    for (int e = 0; e < 32; ++e) atomicAdd(cg + (size_t)(c0 - nx + e) * in, __uint_as_float(r[e]));
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(bDEmpty));
        }
    } else if (warp == kGramLoadWarp) {
        // ------------------------------------------------------------ loader: tokens and raw rows
        const uint64_t pol = policy_evict_last();   // the partner row block reads them again
        uint32_t it = 0, issued = 0;
        bool ok = true;
        for (int w = w0; w < w1 && ok; ++w, ++it) {
            const GramUnit x = gram_unit(L, w);
            const int kv = x.g & 1, jh = x.g >> 1, h = jh % P.Ht, j = jh / P.Ht;
            const uint32_t r = it % (uint32_t)L.raw_slots, ph = (it / (uint32_t)L.raw_slots) & 1;
            if (!W.wait(bar(bREmpty + r), ph ^ 1)) break;
            GramTok* tt = tok_tab((int)r);
            GramTok tk[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int i = lane + 32 * u, tp = x.kb * kGramK + i;
                tk[u] = GramTok{0, 0, 0, 0, -1, 0, 0};
                if (tp < P.T_total) {
                    const TokenInfo ti = resolve_token(P, tp);
                    const bool ok = ti.dst_off >= 0 && ti.hi > ti.lo;
                    const int ps = DIRECT && ok && kv == 0 && P.rs.enabled ? src_pos_of(P, ti.b, ti.lo) : 0;
                    tk[u] = GramTok{ti.b, ti.lo, ti.hi, ti.pt, ti.dst_off, ok, ps};
                }
                tt[i] = tk[u];
            }
            if (DIRECT) {   // the prologue gathers the rows itself
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(bRFull + r));
                continue;
            }
            // the window: from the first token's span start, within its sequence, up to rcap rows
            const int b0 = __shfl_sync(0xffffffffu, tk[0].b, 0), c0 = __shfl_sync(0xffffffffu, tk[0].lo, 0);
            const int ok0 = __shfl_sync(0xffffffffu, tk[0].ok, 0);
            int hm = INT_MIN;
#pragma unroll
            for (int u = 0; u < 2; ++u)
                if (tk[u].ok && tk[u].b == b0) hm = max(hm, tk[u].hi);
            hm = __reduce_max_sync(0xffffffffu, hm);
            const int R = ok0 && hm > c0 ? min(hm - c0, L.rcap) : 0;
            const int n_tgt = __popc(__ballot_sync(0xffffffffu, tk[0].ok)) + __popc(__ballot_sync(0xffffffffu, tk[1].ok));
            if (lane == 0) {
                int* hd = win_hdr((int)r);
                hd[0] = b0;
                hd[1] = c0;
                hd[2] = R;
            }
            __syncwarp();
            const uint32_t bytes = (uint32_t)R * (uint32_t)DS * 2u * (uint32_t)heads + (uint32_t)n_tgt * (uint32_t)dt * 2u;
            if (lane == 0) mbar_arrive_expect_tx(bar(bRFull + r), bytes);
            __syncwarp();
            // source window: one copy per head-block when the rows are contiguous, else one per row
            for (int q = 0; q < heads; ++q) {
                int slot, gs;
                head_block(P, j, h, q, slot, gs);
                const __nv_bfloat16* base = (const __nv_bfloat16*)(kv ? P.src_v[slot] : P.src_k[slot]) +
                                            (long long)b0 * P.sb + (long long)gs * P.sh;
                uint8_t* dstq = src_rows((int)r, q);
                if (P.ss == DS) {
                    if (lane == 0 && R > 0)
                        bulk_g2s(smem_u32(dstq), base + (long long)c0 * P.ss, (uint32_t)R * DS * 2, bar(bRFull + r), pol);
                } else {
                    for (int rr = lane; rr < R; rr += 32)
                        bulk_g2s(smem_u32(dstq + (size_t)rr * L.src_row), base + (long long)(c0 + rr) * P.ss, DS * 2,
                                 bar(bRFull + r), pol);
                }
            }
            // target rows: one copy when the 64 rows are consecutive in a contiguous cache, else one per token
            const __nv_bfloat16* tgt = (const __nv_bfloat16*)(kv ? P.dst_v[j] : P.dst_k[j]);
            const long long hoff = dst_head_off(P, h);
            const long long off0 = __shfl_sync(0xffffffffu, tk[0].dst_off, 0);
            const bool run = __all_sync(0xffffffffu, tk[0].ok && tk[1].ok && tk[0].b == b0 && tk[1].b == b0 &&
                                                         tk[0].dst_off == off0 + (long long)lane * P.dts &&
                                                         tk[1].dst_off == off0 + (long long)(lane + 32) * P.dts) &&
                             !P.paged && P.dts == dt;
            if (run) {
                if (lane == 0)
                    bulk_g2s(smem_u32(tgt_rows((int)r)), tgt + off0 + hoff, (uint32_t)kGramK * dt * 2u, bar(bRFull + r), pol);
            } else {
#pragma unroll
                for (int u = 0; u < 2; ++u)
                    if (tk[u].ok)
                        bulk_g2s(smem_u32(tgt_rows((int)r) + (size_t)(lane + 32 * u) * L.tgt_row),
                                 tgt + tk[u].dst_off + hoff, (uint32_t)dt * 2u, bar(bRFull + r), pol);
            }
            ++issued;
        }
        if (*sAbort) {   // let the copies in flight land before the CTA leaves
            const unsigned long long t0 = globaltimer();
            const uint32_t ns = (uint32_t)L.raw_slots;
            for (uint32_t c = issued > ns ? issued - ns : 0; c < issued; ++c)
                while (!mbar_try_wait(bar(bRFull + c % ns), (c / ns) & 1) && globaltimer() - t0 < kWaitNs) {}
        }
    } else if (DIRECT) {
        // ------------------------------------------------------------ prologue, direct blocks
        // Team `team` of kGramTeamWarps warps takes every kGramTeams-th block.  A thread keeps one
        // chunk pair cp and steps over the block's tokens: per token it copies the pair's two
        // 16-byte chunks of every needed source head and of the target row into their swizzled
        // places, waits for its own copies, and for K un-rotates them in place, with one (cos, sin)
        // per pair for the source heads and, when the two rotations and positions coincide, for
        // the target row as well.
        constexpr int HS = DS / 2;
        constexpr int CPH = DS / 16;
        const int xw = warp - kGramXfWarp0, team = xw / kGramTeamWarps, tw = xw - team * kGramTeamWarps;
        const int cpt = dt / 16, CPM = CPH > cpt ? CPH : cpt;
        const unsigned long long* sTurnS = sTurn;
        const unsigned long long* sTurnT = sTurn + (P.ds >> 1);
        uint32_t it = (uint32_t)team;
        for (int w = w0 + team; w < w1; w += kGramTeams, it += kGramTeams) {
            const GramUnit x = gram_unit(L, w);
            const int kv = x.g & 1, jh = x.g >> 1, h = jh % P.Ht, j = jh / P.Ht;
            const int nh = min(heads, ((x.mb + 1) * 128 + DS - 1) / DS);
            const uint32_t s = it % (uint32_t)L.stages, ph = (it / (uint32_t)L.stages) & 1;
            const uint32_t r = it % (uint32_t)L.raw_slots, rph = (it / (uint32_t)L.raw_slots) & 1;
            if (!W.wait(bar(bZEmpty + s), ph ^ 1)) break;
            if (!W.wait(bar(bRFull + r), rph)) break;
            uint8_t* st = smem + (size_t)s * L.stage_bytes;
            const uint32_t st32 = smem_u32(st);
            const GramTok* tt = tok_tab((int)r);
            const __nv_bfloat16* hb[NHD];
#pragma unroll
            for (int q = 0; q < NHD; ++q) {
                int slot, gs;
                head_block(P, j, h, q, slot, gs);
                hb[q] = (const __nv_bfloat16*)(kv ? P.src_v[slot] : P.src_k[slot]) + (long long)gs * P.sh;
            }
            const __nv_bfloat16* tgt = (const __nv_bfloat16*)(kv ? P.dst_v[j] : P.dst_k[j]) + dst_head_off(P, h);
            // This thread's chunk pair cp for every token i0, i0 + istep, ... of the block: the
            // destination columns (64-channel block and 16-byte chunk within the swizzled row)
            // depend only on cp, a token adds its row offset and the swizzle phase i & 7.
            const uint4 zero = make_uint4(0u, 0u, 0u, 0u);
            // (threads past the last whole stride stay idle: no token is copied or rotated twice)
            const int ttid = tw * 32 + lane, cp = ttid % CPM, istep = kGramTeamWarps * 32 / CPM;
            const int i0 = ttid < istep * CPM ? ttid / CPM : kGramK;
            const bool has_x = cp < CPH, has_y = cp < cpt;
            int c_lo = 0, c_hi = 0, y_lo = 0, y_hi = 0;
            if (has_x) pair_channels(cp * 8, HS, P.rhalf_s, c_lo, c_hi);
            if (has_y) pair_channels(cp * 8, dt >> 1, P.rhalf_t, y_lo, y_hi);
            auto col = [](int c) { return (uint32_t)((c >> 6) * (kGramK * 128)); };
            auto chk = [](int c) { return (uint32_t)((c >> 3) & 7); };
            for (int i = i0; i < kGramK; i += istep) {
                const GramTok tk = tt[i];
                const uint32_t row = (uint32_t)((i >> 3) * 1024 + (i & 7) * 128), x7 = (uint32_t)(i & 7);
                if (has_x) {
                    const long long so = (long long)tk.b * P.sb + (long long)tk.lo * P.ss;
#pragma unroll
                    for (int q = 0; q < NHD; ++q) {
                        if (q >= nh) break;
                        const int cl = q * DS + c_lo, ch = q * DS + c_hi;
                        const uint32_t d_lo = col(cl) + row + ((chk(cl) ^ x7) << 4);
                        const uint32_t d_hi = col(ch) + row + ((chk(ch) ^ x7) << 4);
                        if (tk.ok) {
                            cp_async16(st32 + d_lo, hb[q] + so + c_lo);
                            cp_async16(st32 + d_hi, hb[q] + so + c_hi);
                        } else {
                            *reinterpret_cast<uint4*>(st + d_lo) = zero;
                            *reinterpret_cast<uint4*>(st + d_hi) = zero;
                        }
                    }
                }
                if (has_y) {
                    const uint32_t d_lo = col(in + y_lo) + row + ((chk(in + y_lo) ^ x7) << 4);
                    const uint32_t d_hi = col(in + y_hi) + row + ((chk(in + y_hi) ^ x7) << 4);
                    if (tk.ok) {
                        const __nv_bfloat16* src = tgt + tk.dst_off;
                        cp_async16(st32 + d_lo, src + y_lo);
                        cp_async16(st32 + d_hi, src + y_hi);
                    } else {
                        *reinterpret_cast<uint4*>(st + d_lo) = zero;
                        *reinterpret_cast<uint4*>(st + d_hi) = zero;
                    }
                }
            }
            cp_async_wait_all();
            const bool rot_s = kv == 0 && P.rs.enabled && has_x && cp * 8 < P.rhalf_s;
            const bool rot_t = kv == 0 && P.rt.enabled && has_y && cp * 8 < P.rhalf_t;
            if (rot_s || rot_t) {
                for (int i = i0; i < kGramK; i += istep) {
                    const GramTok tk = tt[i];
                    if (!tk.ok) continue;
                    const uint32_t row = (uint32_t)((i >> 3) * 1024 + (i & 7) * 128), x7 = (uint32_t)(i & 7);
                    float2 cs[8];
                    if (rot_s) {
#pragma unroll
                        for (int e = 0; e < 8; ++e) cs[e] = turn_cs(sTurnS[cp * 8 + e], tk.ps);
#pragma unroll
                        for (int q = 0; q < NHD; ++q) {
                            if (q >= nh) break;
                            const int cl = q * DS + c_lo, ch = q * DS + c_hi;
                            gram_unrotate(st + col(cl) + row + ((chk(cl) ^ x7) << 4),
                                          st + col(ch) + row + ((chk(ch) ^ x7) << 4), cs);
                        }
                    }
                    if (rot_t) {
                        if (!(rot_s && P.rope_same && tk.ps == tk.pt)) {
#pragma unroll
                            for (int e = 0; e < 8; ++e) cs[e] = turn_cs(sTurnT[cp * 8 + e], tk.pt);
                        }
                        gram_unrotate(st + col(in + y_lo) + row + ((chk(in + y_lo) ^ x7) << 4),
                                      st + col(in + y_hi) + row + ((chk(in + y_hi) ^ x7) << 4), cs);
                    }
                }
            }
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(bar(bZFull + s));
                mbar_arrive(bar(bREmpty + r));
            }
        }
    } else {
        // ------------------------------------------------------------ prologue: token-row blocks in shared memory
        // A pass covers a few tokens of the block with the lanes across 16-channel chunk pairs
        // (LX lanes per token for the source head, LY for the target row), so a warp reads whole
        // 128-byte segments of the staged rows and writes whole swizzled rows of the block.
        constexpr int HS = DS / 2;
        constexpr int CPH = DS / 16;                 // chunk pairs (16 channels) per source head
        constexpr int LX = CPH < 32 ? CPH : 32;      // lanes per token, X
        const int xw = warp - kGramXfWarp0;
        const int cpt = dt / 16;                     // chunk pairs of a target row
        const int LY = cpt < 32 ? cpt : 32;          // lanes per token, Y
        const int y_tpp = 32 / LY, y_tok = lane / LY, y_cp = lane % LY;   // per Y pass: tokens, this lane's token and pair
        const unsigned long long* sTurnS = sTurn;
        const unsigned long long* sTurnT = sTurn + (P.ds >> 1);
        uint32_t it = 0;
        for (int w = w0; w < w1; ++w, ++it) {
            const GramUnit x = gram_unit(L, w);
            const int kv = x.g & 1, jh = x.g >> 1, h = jh % P.Ht, j = jh / P.Ht;
            // X head-blocks this row block needs: the rows [0, (mb+1)*128) of the lower triangle
            const int nh = min(heads, ((x.mb + 1) * 128 + DS - 1) / DS);
            const uint32_t s = it % (uint32_t)L.stages, ph = (it / (uint32_t)L.stages) & 1;
            const uint32_t r = it % (uint32_t)L.raw_slots, rph = (it / (uint32_t)L.raw_slots) & 1;
            if (!W.wait(bar(bZEmpty + s), ph ^ 1)) break;
            if (!W.wait(bar(bRFull + r), rph)) break;
            uint8_t* st = smem + (size_t)s * L.stage_bytes;
            const GramTok* tt = tok_tab((int)r);
            const int* hd = win_hdr((int)r);
            const int b0 = hd[0], c0 = hd[1], R = hd[2];
            const bool rot_s = kv == 0 && P.rs.enabled, rot_t = kv == 0 && P.rt.enabled;
            const int xpass = kGramK * LX / 32, ypass = kGramK * LY / 32;
            for (int pc = xw; pc < xpass + ypass; pc += kGramNumXf) {
                if (pc < xpass) {
                    // X: chunk pair cp of every needed source head, span mean of un-rotated rows
                    const int i = pc * (32 / LX) + lane / LX, cp = lane % LX;
                    const GramTok tk = tt[i];
                    int c_lo, c_hi;
                    pair_channels(cp * 8, HS, P.rhalf_s, c_lo, c_hi);
                    const bool rot = rot_s && cp * 8 < P.rhalf_s;
                    float a0[NHD][8], a1[NHD][8];
#pragma unroll
                    for (int q = 0; q < NHD; ++q)
#pragma unroll
                        for (int e = 0; e < 8; ++e) { a0[q][e] = 0.f; a1[q][e] = 0.f; }
                    if (tk.ok) {
                        const bool inwin = tk.b == b0 && tk.lo >= c0 && tk.hi <= c0 + R;
                        for (int sidx = tk.lo; sidx < tk.hi; ++sidx) {
                            float2 cs[8];
                            if (rot) {
                                const int pos = src_pos_of(P, tk.b, sidx);
#pragma unroll
                                for (int e = 0; e < 8; ++e) cs[e] = turn_cs(sTurnS[cp * 8 + e], pos);
                            }
#pragma unroll
                            for (int q = 0; q < NHD; ++q) {
                                if (q >= nh) break;
                                uint4 w0v, w1v;
                                if (inwin) {
                                    const uint8_t* rp = src_rows((int)r, q) + (size_t)(sidx - c0) * L.src_row;
                                    w0v = *reinterpret_cast<const uint4*>(rp + c_lo * 2);
                                    w1v = *reinterpret_cast<const uint4*>(rp + c_hi * 2);
                                } else {
                                    int slot, gs;
                                    head_block(P, j, h, q, slot, gs);
                                    const __nv_bfloat16* rp = (const __nv_bfloat16*)(kv ? P.src_v[slot] : P.src_k[slot]) +
                                                              (long long)tk.b * P.sb + (long long)gs * P.sh +
                                                              (long long)sidx * P.ss;
                                    w0v = __ldg(reinterpret_cast<const uint4*>(rp + c_lo));
                                    w1v = __ldg(reinterpret_cast<const uint4*>(rp + c_hi));
                                }
                                const uint32_t v0[4] = {w0v.x, w0v.y, w0v.z, w0v.w}, v1[4] = {w1v.x, w1v.y, w1v.z, w1v.w};
#pragma unroll
                                for (int e = 0; e < 8; ++e) {
                                    const float x0 = (e & 1) ? bf_hi(v0[e >> 1]) : bf_lo(v0[e >> 1]);
                                    const float x1 = (e & 1) ? bf_hi(v1[e >> 1]) : bf_lo(v1[e >> 1]);
                                    if (rot) {   // R(-theta)
                                        a0[q][e] += fmaf(x0, cs[e].x, x1 * cs[e].y);
                                        a1[q][e] += fmaf(x1, cs[e].x, -x0 * cs[e].y);
                                    } else {
                                        a0[q][e] += x0;
                                        a1[q][e] += x1;
                                    }
                                }
                            }
                        }
                        const float inv = 1.f / (float)(tk.hi - tk.lo);
#pragma unroll
                        for (int q = 0; q < NHD; ++q)
#pragma unroll
                            for (int e = 0; e < 8; ++e) { a0[q][e] *= inv; a1[q][e] *= inv; }
                    }
#pragma unroll
                    for (int q = 0; q < NHD; ++q) {
                        if (q >= nh) break;
                        gram_put(st, i, q * DS + c_lo, q * DS + c_hi, a0[q], a1[q]);
                    }
                } else {
                    // Y: chunk pair cp of the target row, target RoPE undone for K
                    const int yp = pc - xpass;
                    const int i = yp * y_tpp + y_tok, cp = y_cp;
                    const GramTok tk = tt[i];
                    int c_lo, c_hi;
                    pair_channels(cp * 8, dt >> 1, P.rhalf_t, c_lo, c_hi);
                    const bool rot = rot_t && cp * 8 < P.rhalf_t;
                    float y0[8], y1[8];
                    if (tk.ok) {
                        const uint8_t* rp = tgt_rows((int)r) + (size_t)i * L.tgt_row;
                        const uint4 w0v = *reinterpret_cast<const uint4*>(rp + c_lo * 2);
                        const uint4 w1v = *reinterpret_cast<const uint4*>(rp + c_hi * 2);
                        const uint32_t v0[4] = {w0v.x, w0v.y, w0v.z, w0v.w}, v1[4] = {w1v.x, w1v.y, w1v.z, w1v.w};
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            const float u0 = (e & 1) ? bf_hi(v0[e >> 1]) : bf_lo(v0[e >> 1]);
                            const float u1 = (e & 1) ? bf_hi(v1[e >> 1]) : bf_lo(v1[e >> 1]);
                            if (rot) {   // R(-theta)
                                const float2 cs = turn_cs(sTurnT[cp * 8 + e], tk.pt);
                                y0[e] = fmaf(u0, cs.x, u1 * cs.y);
                                y1[e] = fmaf(u1, cs.x, -u0 * cs.y);
                            } else {
                                y0[e] = u0;
                                y1[e] = u1;
                            }
                        }
                    } else {
#pragma unroll
                        for (int e = 0; e < 8; ++e) { y0[e] = 0.f; y1[e] = 0.f; }
                    }
                    gram_put(st, i, in + c_lo, in + c_hi, y0, y1);
                }
            }
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(bar(bZFull + s));
                mbar_arrive(bar(bREmpty + r));
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == kGramMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, 512);
    }
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
            (ds == 64 || ds == 128 || ds == 256) && in / ds <= kGramMaxHeads;
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

template <int DS, int NHD, bool DIRECT>
static cudaError_t launch_gram_tc_v(const TranslateParams& P, const GramLaunch& L, int grid, size_t smem, cudaStream_t s)
{
    // the opt-in is set once per device, so at the largest size any launch asks for
    const cudaError_t e = smem_opt_in<fit_gram_tc_kernel<DS, NHD, DIRECT>>(kSmemMax);
    if (e != cudaSuccess) return e;
    fit_gram_tc_kernel<DS, NHD, DIRECT><<<grid, gram_threads(DIRECT), smem, s>>>(P, L);
    return cudaGetLastError();
}

template <int DS, int NHD>
static cudaError_t launch_gram_tc(const TranslateParams& P, const GramLaunch& L, bool direct, int grid, size_t smem,
                                  cudaStream_t s)
{
    return direct ? launch_gram_tc_v<DS, NHD, true>(P, L, grid, smem, s)
                  : launch_gram_tc_v<DS, NHD, false>(P, L, grid, smem, s);
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
        const int ds = D.src.head_dim;
        GramLaunch L{};
        L.nrows = in + dt;
        L.mbs = in / 128;
        L.nkb = (tgt->total_tokens + kGramK - 1) / kGramK;
        L.kc = L.nkb;   // one unit per (group, row block): one accumulator flush each
        L.nch = L.nkb / L.kc;
        L.units = f->groups * L.nch * L.mbs;
        L.stage_bytes = (unsigned)L.nrows * 128;
        L.src_row = (unsigned)ds * 2;   // rows as in the caches: whole windows move in one copy
        L.tgt_row = (unsigned)dt * 2;
        const unsigned tail = 32 * 8 + (unsigned)(ds / 2 + dt / 2) * 8;   // barriers, flags, turns
        // identity alignment: every span is one source row (or none), gathered by the prologue
        const bool direct = P.span_lo == nullptr;
        bool fits = false;
        if (direct) {   // token tables only in the raw slots; as many block stages as fit
            const unsigned rb = (unsigned)(kGramK * sizeof(GramTok) + 16 + 15) / 16 * 16;
            for (int st = kGramMaxStages; st >= 2 && !fits; --st) {
                L.stages = st;
                L.raw_slots = kGramMaxRaw;
                L.rcap = 0;
                L.raw_bytes = rb;
                L.off_raw = (unsigned)L.stages * L.stage_bytes;
                L.off_bar = L.off_raw + (unsigned)kGramMaxRaw * rb;
                fits = 1024 + L.off_bar + tail <= (unsigned)kSmemMax;
            }
        }
        for (int raw = 2; raw >= 1 && !fits; --raw)
            for (int rcap = 128; rcap >= 64 && !fits; rcap -= 16) {
                const unsigned rb = (unsigned)(kGramK * sizeof(GramTok) + 16 + (size_t)(in / ds) * rcap * L.src_row +
                                               (size_t)kGramK * L.tgt_row + 15) / 16 * 16;
                L.stages = 2;
                L.raw_slots = raw;
                L.rcap = rcap;
                L.raw_bytes = rb;
                L.off_raw = (unsigned)L.stages * L.stage_bytes;
                L.off_bar = L.off_raw + (unsigned)raw * rb;
                fits = 1024 + L.off_bar + tail <= (unsigned)kSmemMax;
            }
        if (!fits) return fit_fail(KVX_ERR_UNSUPPORTED, "fit_accumulate: Gram blocks do not fit shared memory");
        L.lbo = kGramK * 128;   // next 64-channel column block
        L.sbo = 1024;           // next 8-token atom row
        L.G = G;
        L.C = C;
        const long long work = (long long)L.units * L.kc;
        const int grid = (int)(work < f->num_sms ? work : f->num_sms);
        const size_t smem = 1024 + (size_t)L.off_bar + tail;
        cudaError_t ce;
        // in = NHD * ds with in a multiple of 128 and in + dt <= 512
        switch (ds * 8 + in / ds) {
        case 64 * 8 + 2: ce = launch_gram_tc<64, 2>(P, L, direct, grid, smem, s); break;
        case 64 * 8 + 4: ce = launch_gram_tc<64, 4>(P, L, direct, grid, smem, s); break;
        case 64 * 8 + 6: ce = launch_gram_tc<64, 6>(P, L, direct, grid, smem, s); break;
        case 128 * 8 + 1: ce = launch_gram_tc<128, 1>(P, L, direct, grid, smem, s); break;
        case 128 * 8 + 2: ce = launch_gram_tc<128, 2>(P, L, direct, grid, smem, s); break;
        case 128 * 8 + 3: ce = launch_gram_tc<128, 3>(P, L, direct, grid, smem, s); break;
        case 256 * 8 + 1: ce = launch_gram_tc<256, 1>(P, L, direct, grid, smem, s); break;
        default: return fit_fail(KVX_ERR_UNSUPPORTED, "fit_accumulate: no Gram kernel for in %d, d_s %d", in, ds);
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
