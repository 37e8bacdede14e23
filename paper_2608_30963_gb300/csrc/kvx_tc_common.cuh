// kvx_tc_common.cuh -- device helpers shared by the tcgen05 kernels (library-internal):
// PTX wrappers for mbarriers, bulk/tensor copies, TMEM and tcgen05.mma, the
// UMMA shared-memory descriptor, bounded waits and bf16 packing.
#pragma once

#include <atomic>

#include "kvx_common.cuh"

namespace kvx {
namespace {

constexpr int kSmemMax = 232448;                      // 227 KB opt-in shared memory per block

// Dynamic shared memory above 48 KB is a per-device opt-in of each kernel: set it the first time
// the kernel is launched on each device (devices 0..63; others set it on every launch).
template <auto Kernel>
cudaError_t smem_opt_in(int bytes)
{
    static std::atomic<unsigned long long> done{0};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = dev >= 0 && dev < 64 ? 1ull << dev : 0ull;
    if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
    e = cudaFuncSetAttribute(Kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_release);
    return e;
}
constexpr unsigned long long kWaitNs = 1000000000ull;   // bound of every on-chip wait (~1 s)

// ------------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// As above, but the thread may sleep in hardware (up to hint_ns) until the
// phase completes, instead of spinning on the barrier word.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint32_t bar, uint32_t parity, uint32_t hint_ns)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "r"(hint_ns)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ unsigned long long globaltimer()
{
    unsigned long long t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ uint64_t policy_evict_first()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t policy_evict_last()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}
// global -> shared bulk copy completing on an mbarrier (16-byte aligned, size % 16 == 0)
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar, uint64_t pol)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(bar), "l"(pol)
        : "memory");
}
// shared -> global bulk copy in the thread's bulk group
__device__ __forceinline__ void bulk_s2g(void* dst, uint32_t src, uint32_t bytes)
{
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(src), "r"(bytes)
                 : "memory");
}
// Stores one output row of a tile from its staging row (bf16).  The tile holds pair slots
// [a, a + hw) (pair_channels, kvx_common.cuh) of a head of 2 half channels; the staging
// row has the slots' first channels, then their partners.  One bulk copy when the tile is
// the whole row of a fully rotating head; else one per run of consecutive channels (at most
// four).  Every run starts and ends on a multiple of 8 channels (16 bytes).
__device__ __forceinline__ void store_row_slots(__nv_bfloat16* dst, uint32_t srow, int a, int hw, int half, int rhalf)
{
    if (hw == half && rhalf == half) {
        bulk_s2g(dst, srow, (uint32_t)half * 4);
        return;
    }
    const int n_rot = min(max(rhalf - a, 0), hw);   // slots of the tile that are rotating pairs
    if (n_rot > 0) {
        bulk_s2g(dst + a, srow, (uint32_t)n_rot * 2);
        bulk_s2g(dst + a + rhalf, srow + (uint32_t)hw * 2, (uint32_t)n_rot * 2);
    }
    if (n_rot < hw) {
        bulk_s2g(dst + a + n_rot + rhalf, srow + (uint32_t)n_rot * 2, (uint32_t)(hw - n_rot) * 2);
        bulk_s2g(dst + a + n_rot + half, srow + (uint32_t)(hw + n_rot) * 2, (uint32_t)(hw - n_rot) * 2);
    }
}
// The same runs as store_row_slots, written by the calling thread with 16-byte stores (for
// a target cache on another device, written through the peer mapping).
__device__ __forceinline__ void store_row_slots_plain(__nv_bfloat16* dst, const uint8_t* srow, int a, int hw, int half,
                                                      int rhalf)
{
    auto run = [](__nv_bfloat16* d, const uint8_t* s, int n) {
        for (int i = 0; i < n; i += 8) *reinterpret_cast<uint4*>(d + i) = *reinterpret_cast<const uint4*>(s + 2 * i);
    };
    if (hw == half && rhalf == half) {
        run(dst, srow, 2 * half);
        return;
    }
    const int n_rot = min(max(rhalf - a, 0), hw);
    if (n_rot > 0) {
        run(dst + a, srow, n_rot);
        run(dst + a + rhalf, srow + hw * 2, n_rot);
    }
    if (n_rot < hw) {
        run(dst + a + n_rot + rhalf, srow + n_rot * 2, hw - n_rot);
        run(dst + a + n_rot + half, srow + (hw + n_rot) * 2, hw - n_rot);
    }
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait0() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// 16-byte asynchronous copy global -> shared by the issuing thread (cached in L2 only); the thread
// waits for its own copies with cp_async_wait_all().
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all()
{
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void fence_mbar_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }

// Programmatic dependent launch: wait until the grids this launch depends on have
// completed and their memory is visible; allow the next dependent launch to begin.
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish()
{
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem] . B[smem]^T, bf16 inputs, fp32 accumulate
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&r)[8])
{
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row atoms 1024 B apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);      // start address
    d |= (uint64_t)1 << 16;                         // leading byte offset (unused for swizzled K-major)
    d |= (uint64_t)(1024u >> 4) << 32;              // stride byte offset between 8-row atoms
    d |= (uint64_t)1 << 46;                         // descriptor version
    d |= (uint64_t)2 << 61;                         // 128-byte swizzle
    return d;
}

// Byte offset of element (row, k) in a K-major SW128 tile with `rows` rows
// (K split into 64-element blocks of rows*128 bytes).
__device__ __forceinline__ uint32_t sw128_off(int row, int k, int rows)
{
    const int kb = k >> 6, c = (k >> 3) & 7, e = k & 7;
    return (uint32_t)(kb * rows * 128 + (row >> 3) * 1024 + (row & 7) * 128 + ((c ^ (row & 7)) << 4) + e * 2);
}

// ------------------------------------------------------------------ bounded waits
struct Waiter {
    volatile int* abort;
    unsigned* status;
    unsigned long long limit_ns = kWaitNs;   // bound of each wait
    __device__ __forceinline__ bool wait(uint32_t bar, uint32_t parity) const
    {
        if (mbar_try_wait(bar, parity)) return true;
        const unsigned long long t0 = globaltimer();
        while (true) {
            if (mbar_try_wait_sleep(bar, parity, 100000u)) return true;
            if (*abort) return false;
            if (globaltimer() - t0 > limit_ns) {
                *abort = 1;
                set_status(status, KVX_DEV_WAIT_TIMEOUT);
                return false;
            }
        }
    }
};

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ uint32_t pack_bf16(float a, float b)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&v);
}

// Undo a rotation on one rotary pair (x0 from the first half, x1 from the second):
//   u0 = x0 cos + x1 sin,  u1 = x1 cos - x0 sin,
// evaluated as fma(x0, cos, x1 sin) and fma(x1, cos, -(x0 sin)), the order the
// identity-alignment kernel uses, so the two kernels agree bit for bit on
// single-token spans.
__device__ __forceinline__ void unrotate1(float x0, float x1, float2 cs, float& u0, float& u1)
{
    u0 = fmaf(x0, cs.x, x1 * cs.y);
    u1 = fmaf(x1, cs.x, -x0 * cs.y);
}
// The same, accumulated onto (a0, a1) for the later rows of a span:
// a0 = fma(x1, sin, fma(x0, cos, a0)), a1 = fma(x0, -sin, fma(x1, cos, a1)).
__device__ __forceinline__ void unrotate_acc(float x0, float x1, float2 cs, float& a0, float& a1)
{
    a0 = fmaf(x1, cs.y, fmaf(x0, cs.x, a0));
    a1 = fmaf(x0, -cs.y, fmaf(x1, cs.x, a1));
}

// Apply a rotation to one rotary pair:  y0 = x0 cos - x1 sin,  y1 = x1 cos + x0 sin,
// evaluated as fma(x0, cos, -(x1 sin)) and fma(x1, cos, x0 sin), as in the
// identity-alignment kernel's epilogue.
__device__ __forceinline__ void rotate1(float x0, float x1, float2 cs, float& y0, float& y1)
{
    const float a = x0, b = x1;
    y0 = fmaf(a, cs.x, -b * cs.y);
    y1 = fmaf(b, cs.x, a * cs.y);
}

// The fp32 of two 8-column TMEM loads (columns c..c+7 of the first and second
// rotary halves) rotated by cs[0..7] (rot) and rounded to bf16: out0 = first half,
// out1 = second half.
__device__ __forceinline__ void rotate8_to_bf16(const uint32_t (&r0)[8], const uint32_t (&r1)[8], const float2 (&cs)[8],
                                                bool rot, uint4& out0, uint4& out1)
{
    float y0[8], y1[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        y0[e] = __uint_as_float(r0[e]);
        y1[e] = __uint_as_float(r1[e]);
        if (rot) rotate1(y0[e], y1[e], cs[e], y0[e], y1[e]);
    }
    out0 = make_uint4(pack_bf16(y0[0], y0[1]), pack_bf16(y0[2], y0[3]), pack_bf16(y0[4], y0[5]), pack_bf16(y0[6], y0[7]));
    out1 = make_uint4(pack_bf16(y1[0], y1[1]), pack_bf16(y1[2], y1[3]), pack_bf16(y1[4], y1[5]), pack_bf16(y1[6], y1[7]));
}

// PP consecutive bf16 values (PP in {1,2,4}) as one raw load.
template <int PP> struct Raw;
template <> struct Raw<4> { using T = uint2; };
template <> struct Raw<2> { using T = uint32_t; };
template <> struct Raw<1> { using T = unsigned short; };

template <int PP>
__device__ __forceinline__ typename Raw<PP>::T load_raw(const __nv_bfloat16* p)
{
    return *reinterpret_cast<const typename Raw<PP>::T*>(p);
}
__device__ __forceinline__ void unpack(uint2 w, float (&x)[4])
{
    x[0] = bf_lo(w.x); x[1] = bf_hi(w.x); x[2] = bf_lo(w.y); x[3] = bf_hi(w.y);
}
__device__ __forceinline__ void unpack(uint32_t w, float (&x)[2]) { x[0] = bf_lo(w); x[1] = bf_hi(w); }
__device__ __forceinline__ void unpack(unsigned short w, float (&x)[1]) { x[0] = __uint_as_float((uint32_t)w << 16); }

template <int PP>
__device__ __forceinline__ void store_bf16_smem(uint8_t* p, const float (&x)[PP])
{
    if constexpr (PP == 4) {
        *reinterpret_cast<uint2*>(p) = make_uint2(pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]));
    } else if constexpr (PP == 2) {
        *reinterpret_cast<uint32_t*>(p) = pack_bf16(x[0], x[1]);
    } else {
        __nv_bfloat16 v = __float2bfloat16_rn(x[0]);
        *reinterpret_cast<__nv_bfloat16*>(p) = v;
    }
}

}  // namespace
}  // namespace kvx
