// kvx_tc_aligned.cu -- tensor-core translation kernel for identity token alignment.
//
// When the source and target tokenisations coincide (span of target token t is
// source token t, the within-family handoff of paper Section 6.2), the A operand
// of the projection is the source cache itself: row t of the tile is the
// concatenation of the grouped source heads at token t, un-rotated for K.  The
// kernel therefore loads A straight into the UMMA K-major 128-byte-swizzled
// layout with tensor-TMA boxes (one box = [128 tokens x 64 channels] of one
// head = one K-block of A), un-rotates K tiles in place, and feeds the tensor
// core from those buffers.  V tiles need no prologue work at all.
//
// Persistent, one CTA per SM.  Work unit = (group, tile) with group = (target
// layer j, target head h, K|V, output split nt) and tiles of 128 tokens laid
// per sequence.  K-blocks stream through a ring of NS slots:
//   warp 0 (lane 0)  producer: B image per group (bulk copy), A K-blocks (tensor TMA)
//   warp 1           MMA: TMEM allocation, tcgen05.mma per K-block, commits
//   warps 2-9        epilogue: TMEM -> target RoPE -> bf16 -> cache (bulk stores);
//                    two warps per TMEM lane quadrant, each taking half of the RoPE pairs
//   warps 10-17      prologue: in-place source-RoPE undo of K tiles
// Every wait is bounded (~1 s, then KVX_DEV_WAIT_TIMEOUT and a drained exit).
#include <cuda.h>
#include <stddef.h>
#include <string.h>

#include "kvx_common.cuh"
#include "kvx_kernels.h"
#include "kvx_schedule.h"
#include "kvx_tc_common.cuh"

namespace kvx {
namespace {

constexpr int kTileM = 128;
constexpr int kBlockK = 64;                       // channels per K-block (one 128-byte swizzle row)
constexpr int kBlockBytes = kTileM * kBlockK * 2;  // 16 KB
constexpr int kMaxSlots = 16;
constexpr int kProducerWarp = 0;
constexpr int kMmaWarp = 1;
constexpr int kEpiWarp0 = 2;
constexpr int kNumEpiWarps = 8;                    // two per TMEM lane quadrant, splitting the columns
constexpr int kXfWarp0 = kEpiWarp0 + kNumEpiWarps;
constexpr int kNumXfWarps = 8;
constexpr int kXfThreads = kNumXfWarps * 32;
constexpr int kThreads = (kXfWarp0 + kNumXfWarps) * 32;

// barrier indices
constexpr int kBarBFull = 0, kBarBEmpty = 1;
constexpr int kBarDFull = 2;                        // +buf (2)
constexpr int kBarDEmpty = 4;                       // +buf (2)
constexpr int kBarFull = 6;                         // +slot: TMA landed
constexpr int kBarEmpty = kBarFull + kMaxSlots;     // +slot: MMA done with it
// +(K tile % nkready): every K-block of that K tile has been un-rotated.  At most
// nslots/nblk + 1 K tiles sit between "rotated" and "consumed by the MMA" (the
// slot ring bounds it), so a ring of nkready = nslots/nblk + 2 barriers never
// completes one twice before the MMA has waited on it.
constexpr int kBarKReady = kBarEmpty + kMaxSlots;
constexpr int kMaxKReady = kMaxSlots + 2;
// +quad*2 + {0,1}: the two epilogue warps of a TMEM lane quadrant meet here before
// writing the shared staging rows (0) and before storing them (1)
constexpr int kBarPair = kBarKReady + kMaxKReady;
// +buf: the epilogue has read the (cos, sin) the prologue left in TMEM for a K tile
constexpr int kBarCsFree = kBarPair + 8;
// after an abort: every MMA the issuer started has completed (before TMEM is freed)
constexpr int kBarMmaDone = kBarCsFree + 2;
constexpr int kNumBars = kBarMmaDone + 1;

struct AlignedParams {
    // geometry
    int Hs, ds, Ht, dt, in_dim, r, e, dense, Lt;
    int n_tile, n_split, groups, nblk, nslots, nkready, m_tiles_max;
    // source
    int batch, src_max_seq;
    const int* src_seq_len;
    const int* src_pos;
    // target
    int T_total;
    const int* seq_off;
    const int* tgt_pos;
    int paged, dst_max_seq;
    long long db, dh, dts;
    const int* page_table;
    int max_pages, page_size, num_pages;
    RopeTable rs, rt;
    int max_position;
    int plain_stores;   // target rows written with 16-byte thread stores (a peer device's cache)
    unsigned long long wait_ns;   // bound of each wait (0: ~1 s)
    int stall_unit1;              // diagnostics: CTA 0's producer stops before its (stall_unit1 - 1)-th unit with rows
    unsigned* status;
    const void* w;
    unsigned idesc, tmem_cols, b_bytes, stage_row_bytes;
    // When source and target rotations coincide (same base, head_dim and positions), the prologue
    // leaves each K tile's (cos, sin) in TMEM columns [cs_col + buf*d, +d) for the epilogue.
    int share_cs;
    unsigned cs_col;
    unsigned off_b, off_ring, off_stage, off_bar, off_misc, off_seq;
    // rotation turns (kvx_common.cuh): source [0, ds/2), target [128, 128 + dt/2); read
    // warp-uniformly, so from the constant bank rather than shared memory
    unsigned long long turns[256];
    void* dst_k[KVX_MAX_ALIGNED_LAYERS];
    void* dst_v[KVX_MAX_ALIGNED_LAYERS];
    CUtensorMap maps[2 * KVX_MAX_ALIGNED_LAYERS];   // [j*2 + kv]: source K/V of target layer j
    // V share of each CTA (an index of the same equal split as the K shares), chosen on the host
    // so that CTAs with a costly K share get a cheap V share; unused above kMaxVmap CTAs
    int use_vmap;
    unsigned short vmap[256];
};
constexpr int kMaxVmap = 256;

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap* map, int c0, int c1, int c2, int c3,
                                            uint32_t bar, uint64_t pol)
{
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%2, %3, %4, %5}], [%6], %7;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar), "l"(pol)
        : "memory");
}

static_assert(sizeof(AlignedParams) <= 32764, "kernel parameter space");

struct AUnit {
    int j, h, kv, nt, g;
    int b, t0, rows;   // sequence, first token, valid rows (0: no such tile)
};

// Iterates a CTA's units in order with counters only (no divisions per unit):
// its share of K units, then its share of V units; each share group-major.
struct Walker {
    int count, n1, it;   // n1: units of the first share
    int kv1;             // K|V of the first share
    int kv, j, h, nt, k, b;
    int u0, v0, m_tiles, n_split, Ht, batch;
    const int* tile_off;
    const int* seq_off;
    AUnit x;

    __device__ __forceinline__ void fill()
    {
        x.j = j; x.h = h; x.kv = kv; x.nt = nt;
        x.g = ((j * Ht + h) * 2 + kv) * n_split + nt;
        if (k >= tile_off[batch]) { x.b = 0; x.t0 = 0; x.rows = 0; return; }
        while (b + 1 < batch && tile_off[b + 1] <= k) ++b;
        x.b = b;
        x.t0 = (k - tile_off[b]) * kTileM;
        x.rows = min(kTileM, seq_off[b + 1] - seq_off[b] - x.t0);
    }
    __device__ __forceinline__ void seek(int idx, int kv_)
    {
        kv = kv_;
        const int hg = idx / m_tiles;
        k = idx - hg * m_tiles;
        nt = hg % n_split;
        const int jh = hg / n_split;
        h = jh % Ht;
        j = jh / Ht;
        b = 0;
        fill();
    }
    // K units [u0, u1) and V units [v0, v1) of the per-K|V unit index space; the V share first
    // when v_first, else the K share first
    __device__ __forceinline__ void start(int u0_, int u1_, int v0_, int v1_, const AlignedParams& P,
                                          const int* tile_off_, const int* seq_off_, bool v_first)
    {
        kv1 = v_first ? 1 : 0;
        u0 = v_first ? v0_ : u0_;   // first share
        v0 = v_first ? u0_ : v0_;   // second share
        n1 = v_first ? v1_ - v0_ : u1_ - u0_;
        count = (u1_ - u0_) + (v1_ - v0_);
        it = 0;
        m_tiles = P.m_tiles_max; n_split = P.n_split; Ht = P.Ht; batch = P.batch;
        tile_off = tile_off_; seq_off = seq_off_;
        if (n1 > 0) seek(u0, kv1);
        else if (count > 0) seek(v0, kv1 ^ 1);
    }
    __device__ __forceinline__ bool more() const { return it < count; }
    __device__ __forceinline__ void next()
    {
        if (++it >= count) return;
        if (it == n1) { seek(v0, kv1 ^ 1); return; }
        if (++k == m_tiles) {
            k = 0;
            b = 0;
            if (++nt == n_split) {
                nt = 0;
                if (++h == Ht) { h = 0; ++j; }
            }
        }
        fill();
    }
    // no later unit of this CTA uses the current group's weights
    __device__ __forceinline__ bool last_of_group() const
    {
        return it + 1 == count || it + 1 == n1 || k + 1 >= tile_off[batch];
    }
};

// position in the K-block slot ring
struct SlotPos {
    uint32_t idx, phase;
    __device__ __forceinline__ void adv(uint32_t n)
    {
        if (++idx == n) { idx = 0; phase ^= 1; }
    }
};

// HS: half head_dim of the source (32, 64 or 128).  VAR: 0 = the normal kernel; 1 = with the
// diagnostics of the bounded waits (a wait bound other than ~1 s, a stalled producer); 2 = target
// rows written with thread stores (a target cache on another device).
template <int HS, int VAR>
__global__ void __launch_bounds__(kThreads, 1) translate_tc_aligned_kernel(const __grid_constant__ AlignedParams P)
{
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // 1024-byte aligned base, derived from smem_raw by pointer arithmetic so that the
    // compiler keeps every access below in the shared address space
    const uint32_t pad = (1024u - (smem_u32(smem_raw) & 1023u)) & 1023u;
    uint8_t* smem = smem_raw + pad;
    uint8_t* sB = smem + P.off_b;
    uint8_t* sRing = smem + P.off_ring;
    uint8_t* sStage = smem + P.off_stage;
    uint64_t* sBar = reinterpret_cast<uint64_t*>(smem + P.off_bar);
    volatile int* sAbort = reinterpret_cast<volatile int*>(smem + P.off_misc);
    uint32_t* sTmemBase = reinterpret_cast<uint32_t*>(smem + P.off_misc + 4);
    int* sSeqOff = reinterpret_cast<int*>(smem + P.off_seq);            // [batch+1]
    int* sSrcLen = sSeqOff + (P.batch + 1);                              // [batch]
    int* sTileOff = sSrcLen + P.batch;                                   // [batch+1]
    const unsigned long long* sTurnS = P.turns;
    const unsigned long long* sTurnT = P.turns + 128;
    // K-block slots: as many as fit after the fixed regions, given the actual alignment of the
    // dynamic shared memory base (the host sized P.nslots for a 1024-byte-aligned base)
    const uint32_t fit = ((uint32_t)kSmemMax - pad - P.off_ring) / kBlockBytes;
    const uint32_t NS = fit < (uint32_t)P.nslots ? fit : (uint32_t)P.nslots;
    const uint32_t NKR = NS / P.nblk + 2;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    auto bar = [&](int i) { return (uint32_t)__cvta_generic_to_shared(&sBar[i]); };

    // On-chip set-up first (barriers, TMEM): with programmatic dependent launch it
    // overlaps the tail of the previous kernel in the stream.
    if (threadIdx.x == 0) {
        *sAbort = 0;
        mbar_init(bar(kBarBFull), 1);
        mbar_init(bar(kBarBEmpty), 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(kBarDFull + i), 1);
            mbar_init(bar(kBarDEmpty + i), kNumEpiWarps);
        }
        for (uint32_t i = 0; i < NS; ++i) {
            mbar_init(bar(kBarFull + i), 1);
            mbar_init(bar(kBarEmpty + i), 2);   // the MMA's commit and the prologue's release
        }
        for (uint32_t i = 0; i < NKR; ++i) mbar_init(bar(kBarKReady + i), kNumXfWarps);
        for (int i = 0; i < 8; ++i) mbar_init(bar(kBarPair + i), 2);
        for (int i = 0; i < 2; ++i) mbar_init(bar(kBarCsFree + i), kNumEpiWarps);
        mbar_init(bar(kBarMmaDone), 1);
        fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        tmem_alloc((uint32_t)__cvta_generic_to_shared(sTmemBase), P.tmem_cols);
        tmem_relinquish();
    }
    // Nothing above touched global memory.  Every access below may read what an
    // earlier kernel in the stream wrote (or overwrite what it reads), so wait for it.
    grid_dependency_wait();
    grid_launch_dependents();
    for (int i = threadIdx.x; i <= P.batch; i += blockDim.x) sSeqOff[i] = __ldg(&P.seq_off[i]);
    for (int i = threadIdx.x; i < P.batch; i += blockDim.x) sSrcLen[i] = __ldg(&P.src_seq_len[i]);
    __syncthreads();
    if (threadIdx.x == 0) {   // per-sequence tile offsets
        int acc = 0;
        for (int b = 0; b < P.batch; ++b) {
            sTileOff[b] = acc;
            const int T = sSeqOff[b + 1] - sSeqOff[b];
            acc += T > 0 ? (T + kTileM - 1) / kTileM : 0;
        }
        sTileOff[P.batch] = acc;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *sTmemBase;

    constexpr bool DIAG = VAR == 1, PLAIN = VAR == 2;
    const Waiter W{sAbort, P.status, DIAG && P.wait_ns ? P.wait_ns : kWaitNs};
    // Work split: each CTA takes an equal share of the K units and of the V units
    // (K units cost more: the source RoPE undo).  Even CTAs walk their V share first and
    // odd CTAs their K share first, so that at any time about half the SMs run K tiles
    // (bound by the un-rotation) and half V tiles (bound by HBM).  Within each share
    // units run group-major, so a group's weight tile stays resident.
    const bool v_first = (blockIdx.x & 1) == 0;
    const int hgroups = P.groups / 2;                          // (j, h, nt) per K|V
    const long long UH = (long long)hgroups * P.m_tiles_max;
    const int u0 = (int)((long long)blockIdx.x * UH / gridDim.x);
    const int u1 = (int)((long long)(blockIdx.x + 1) * UH / gridDim.x);
    // the V share mirrors the CTA order, so a CTA with one K unit more gets one V unit fewer
    const int vr = P.use_vmap ? (int)P.vmap[blockIdx.x] : (int)gridDim.x - 1 - (int)blockIdx.x;
    const int v0 = (int)((long long)vr * UH / gridDim.x);
    const int v1 = (int)((long long)(vr + 1) * UH / gridDim.x);
    const int blk_per_head = (2 * HS) / kBlockK;       // K-blocks of one source head
    const int hw = P.n_tile >> 1;

    if (warp == kProducerWarp) {
        // ------------------------------------------------------------ producer (one thread)
        if (lane == 0) {
            const uint64_t pol_stream = policy_evict_first();
            const uint64_t pol_keep = policy_evict_last();
            int cur_g = -1;
            uint32_t b_loads = 0, slot_cnt = 0;
            SlotPos sp{0, 0};
            bool ok = true;
            int nunit = 0;   // units with rows walked so far
            Walker wk;
            for (wk.start(u0, u1, v0, v1, P, sTileOff, sSeqOff, v_first); wk.more(); wk.next()) {
                const AUnit& x = wk.x;
                if (x.rows <= 0) continue;
                if (DIAG && blockIdx.x == 0 && ++nunit == P.stall_unit1) {
                    // diagnostics: a copy that never comes; the consumers' bounded waits run out
                    const unsigned long long t0 = globaltimer();
                    while (!*sAbort && globaltimer() - t0 < 4 * W.limit_ns) {}
                    break;
                }
                // A K-blocks first: they do not depend on the weights, so at a group switch the
                // ring refills while the previous group's last tiles drain
                const CUtensorMap* map = &P.maps[x.j * 2 + x.kv];
                const int g0 = P.dense ? 0 : (P.r > 1 ? x.h * P.r : x.h / P.e);
                for (int kb = 0; kb < P.nblk; ++kb) {
                    const uint32_t slot = sp.idx;
                    if (!W.wait(bar(kBarEmpty + slot), sp.phase ^ 1)) { ok = false; break; }
                    mbar_arrive_expect_tx(bar(kBarFull + slot), kBlockBytes);
                    tma_load_4d((uint32_t)__cvta_generic_to_shared(sRing) + slot * kBlockBytes, map,
                                (kb % blk_per_head) * kBlockK, x.t0, g0 + kb / blk_per_head, x.b,
                                bar(kBarFull + slot), pol_stream);
                    ++slot_cnt;
                    sp.adv(NS);
                }
                if (!ok) break;
                if (x.g != cur_g) {
                    if (!W.wait(bar(kBarBEmpty), (b_loads & 1) ^ 1)) { ok = false; break; }
                    mbar_arrive_expect_tx(bar(kBarBFull), P.b_bytes);
                    const uint8_t* img = (const uint8_t*)P.w + (size_t)x.g * P.b_bytes;
                    const uint32_t piece = P.b_bytes / 4;
                    for (int q = 0; q < 4; ++q)
                        bulk_g2s((uint32_t)__cvta_generic_to_shared(sB) + q * piece, img + (size_t)q * piece, piece,
                                 bar(kBarBFull), pol_keep);
                    ++b_loads;
                    cur_g = x.g;
                }
                if (!ok) break;
            }
            if (*sAbort) {   // let copies in flight land before leaving
                const unsigned long long t0 = globaltimer();
                for (uint32_t c = slot_cnt > NS ? slot_cnt - NS : 0; c < slot_cnt; ++c)
                    while (!mbar_try_wait(bar(kBarFull + c % NS), (c / NS) & 1) &&
                           globaltimer() - t0 < W.limit_ns) {}
                if (b_loads)
                    while (!mbar_try_wait(bar(kBarBFull), (b_loads - 1) & 1) && globaltimer() - t0 < W.limit_ns) {}
            }
        }
        __syncwarp();
    } else if (warp == kMmaWarp) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            int cur_g = -1;
            uint32_t b_cnt = 0, tcount = 0;
            SlotPos sp{0, 0};
            uint32_t kr_idx = 0, kr_phase = 0;
            bool ok = true;
            Walker wk;
            for (wk.start(u0, u1, v0, v1, P, sTileOff, sSeqOff, v_first); wk.more(); wk.next()) {
                const AUnit& x = wk.x;
                if (x.rows <= 0) continue;
                if (x.g != cur_g) {
                    if (!W.wait(bar(kBarBFull), b_cnt & 1)) break;
                    ++b_cnt;
                    cur_g = x.g;
                }
                const bool rot = x.kv == 0 && P.rs.enabled;
                const uint32_t buf = tcount & 1;
                if (!W.wait(bar(kBarDEmpty + buf), ((tcount >> 1) & 1) ^ 1)) break;
                const uint32_t d = tmem_base + buf * (uint32_t)P.n_tile;
                const uint32_t b0 = (uint32_t)__cvta_generic_to_shared(sB);
                if (rot) {   // K tile: wait until the prologue has un-rotated all its K-blocks
                    if (!W.wait(bar(kBarKReady + kr_idx), kr_phase)) break;
                    if (++kr_idx == NKR) { kr_idx = 0; kr_phase ^= 1; }
                }
                for (int kb = 0; kb < P.nblk; ++kb) {
                    const uint32_t slot = sp.idx;
                    const uint32_t par = sp.phase;
                    if (!rot && !W.wait(bar(kBarFull + slot), par)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t a0 = (uint32_t)__cvta_generic_to_shared(sRing) + slot * kBlockBytes;
#pragma unroll
                    for (int kk = 0; kk < kBlockK / 16; ++kk) {
                        const uint64_t ad = sw128_desc(a0 + kk * 32);
                        const uint64_t bd = sw128_desc(b0 + kb * (P.n_tile * 128) + kk * 32);
                        umma_bf16(d, ad, bd, P.idesc, (kb > 0 || kk > 0) ? 1u : 0u);
                    }
                    umma_commit(bar(kBarEmpty + slot));
                    sp.adv(NS);
                }
                if (!ok) break;
                umma_commit(bar(kBarDFull + buf));
                // the last valid tile of this group in the CTA's range releases B
                const bool last = wk.last_of_group();
                if (last) umma_commit(bar(kBarBEmpty));
                ++tcount;
            }
            if (*sAbort) {   // MMAs whose results nobody waited for must finish before TMEM is freed
                umma_commit(bar(kBarMmaDone));
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(bar(kBarMmaDone), 0) && globaltimer() - t0 < W.limit_ns) {}
            }
        }
        __syncwarp();
    } else if (warp < kEpiWarp0 + kNumEpiWarps) {
        // ------------------------------------------------------------ epilogue
        const int quad = warp & 3;
        const int half = (warp - kEpiWarp0) >> 2;          // which half of the RoPE pairs
        const int m = quad * 32 + lane;
        const int pc_begin = half * (hw >> 1), pc_end = pc_begin + (hw >> 1);
        uint8_t* srow = sStage + (size_t)m * P.stage_row_bytes;
        const uint32_t srow_u32 = (uint32_t)__cvta_generic_to_shared(srow);
        uint32_t tcount = 0, kc = 0;   // kc: K tiles seen (selects the shared (cos, sin) buffer)
        Walker wk;
        for (wk.start(u0, u1, v0, v1, P, sTileOff, sSeqOff, v_first); wk.more(); wk.next()) {
            const AUnit& x = wk.x;
            if (x.rows <= 0) continue;
            const uint32_t buf = tcount & 1;
            // output row of this thread, resolved while the tile is computed
            const int t = x.t0 + m;
            bool valid = m < x.rows;
            long long dst_off = -1;
            int pt = 0;
            if (valid) {
                int S = sSrcLen[x.b];
                if (S > P.src_max_seq) S = P.src_max_seq;
                if (t >= S) { set_status(P.status, KVX_DEV_SPAN_CLAMPED); valid = false; }
                const int p = P.tgt_pos ? __ldg(&P.tgt_pos[sSeqOff[x.b] + t]) : t;
                pt = P.rt.enabled ? clamp_pos(p, P.max_position, P.status) : 0;
                if (!P.paged) {
                    if (t >= P.dst_max_seq) { set_status(P.status, KVX_DEV_SEQ_CLAMPED); valid = false; }
                    else dst_off = (long long)x.b * P.db + (long long)t * P.dts;
                } else {
                    const int pi = t / P.page_size;
                    const int page = pi < P.max_pages ? __ldg(&P.page_table[(size_t)x.b * P.max_pages + pi]) : -1;
                    if (page < 0 || page >= P.num_pages) { set_status(P.status, KVX_DEV_PAGE_INVALID); valid = false; }
                    else dst_off = ((long long)page * P.page_size + (t % P.page_size)) * (long long)P.Ht * P.dt;
                }
            }
            const bool rot = x.kv == 0 && P.rt.enabled;
            if (!W.wait(bar(kBarDFull + buf), (tcount >> 1) & 1)) break;
            tc_fence_after();
            // the staging row is shared by the two warps of this quadrant; the row's
            // previous store (issued by the thread of lane parity = half) must have read it
            bulk_wait_read0();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kBarPair + quad * 2));
            if (!W.wait(bar(kBarPair + quad * 2), tcount & 1)) break;
            const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + buf * (uint32_t)P.n_tile;
            const bool shared_cs = rot && P.share_cs;          // (cos, sin) left in TMEM by the prologue
            const uint32_t cs_addr = tmem_base + ((uint32_t)(quad * 32) << 16) + P.cs_col + (kc & 1) * (uint32_t)P.dt;
            for (int pc = pc_begin; pc < pc_end; pc += 8) {
                uint32_t r0[8], r1[8];
                tmem_ld8(taddr + pc, r0);
                tmem_ld8(taddr + hw + pc, r1);
                float2 cs[8];
                if (shared_cs) {
                    uint32_t v[16];
                    tmem_ld16(cs_addr + 2 * (x.nt * hw + pc), v);
                    tmem_ld_wait();
#pragma unroll
                    for (int e2 = 0; e2 < 8; ++e2) cs[e2] = make_float2(__uint_as_float(v[2 * e2]), __uint_as_float(v[2 * e2 + 1]));
                } else if (rot) {
#pragma unroll
                    for (int e2 = 0; e2 < 8; ++e2) cs[e2] = turn_cs(sTurnT[x.nt * hw + pc + e2], pt);
                }
                tmem_ld_wait();
                float y0[8], y1[8];
#pragma unroll
                for (int e2 = 0; e2 < 8; ++e2) { y0[e2] = __uint_as_float(r0[e2]); y1[e2] = __uint_as_float(r1[e2]); }
                if (rot) {
#pragma unroll
                    for (int e2 = 0; e2 < 8; ++e2) {
                        const float a = y0[e2], bb = y1[e2];
                        y0[e2] = fmaf(a, cs[e2].x, -bb * cs[e2].y);
                        y1[e2] = fmaf(bb, cs[e2].x, a * cs[e2].y);
                    }
                }
                *reinterpret_cast<uint4*>(srow + pc * 2) =
                    make_uint4(pack_bf16(y0[0], y0[1]), pack_bf16(y0[2], y0[3]), pack_bf16(y0[4], y0[5]),
                               pack_bf16(y0[6], y0[7]));
                *reinterpret_cast<uint4*>(srow + (hw + pc) * 2) =
                    make_uint4(pack_bf16(y1[0], y1[1]), pack_bf16(y1[2], y1[3]), pack_bf16(y1[4], y1[5]),
                               pack_bf16(y1[6], y1[7]));
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(bar(kBarDEmpty + buf));
                if (shared_cs) mbar_arrive(bar(kBarCsFree + (kc & 1)));
            }
            if (x.kv == 0) ++kc;
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kBarPair + quad * 2 + 1));
            if (!W.wait(bar(kBarPair + quad * 2 + 1), tcount & 1)) break;
            if ((lane & 1) == half && valid && dst_off >= 0) {   // the quadrant's rows, split between its two warps
                __nv_bfloat16* dst = (__nv_bfloat16*)(x.kv ? P.dst_v[x.j] : P.dst_k[x.j]) + dst_off +
                                     (P.paged ? (long long)x.h * P.dt : (long long)x.h * P.dh);
                if (PLAIN) {
                    store_row_slots_plain(dst, srow, x.nt * hw, hw, P.dt >> 1, P.dt >> 1);
                } else if (P.n_split == 1) {
                    bulk_s2g(dst, srow_u32, (uint32_t)P.dt * 2);
                } else {
                    bulk_s2g(dst + x.nt * hw, srow_u32, (uint32_t)hw * 2);
                    bulk_s2g(dst + (P.dt >> 1) + x.nt * hw, srow_u32 + hw * 2, (uint32_t)hw * 2);
                }
                if (!PLAIN) bulk_commit();
            }
            ++tcount;
        }
        bulk_wait0();
    } else {
        // ------------------------------------------------------------ prologue: undo source RoPE in place
        // Thread layout over a K tile: thread = token row = TMEM lane of its warp's
        // quadrant (row = 32*(warp%4) + lane), and the two warps of a quadrant split
        // the rotary pairs (i, i+HS).  Each (cos, sin) is computed once for all
        // grouped heads.  Pairs go 8 at a time (one 16-byte chunk of each half); under
        // the 128-byte swizzle the 8 rows of a shared-memory phase hit distinct banks.
        const int xt = threadIdx.x - kXfWarp0 * 32;
        const int row = (warp & 3) * 32 + lane;
        const int part = (warp - kXfWarp0) >> 2;          // 0 or 1
        const int heads = P.in_dim / (2 * HS);            // heads in one A row
        constexpr int kChunks = HS / 8;                    // 16-byte chunks per half head
        constexpr int kMine = kChunks / 2;                 // chunks per thread
        const uint32_t cs_lane = tmem_base + ((uint32_t)((warp & 3) * 32) << 16) + P.cs_col;
        SlotPos sp{0, 0};
        uint32_t kr_idx = 0, kc = 0;
        bool ok = true;
        Walker wk;
        for (wk.start(u0, u1, v0, v1, P, sTileOff, sSeqOff, v_first); wk.more(); wk.next()) {
            const AUnit& x = wk.x;
            if (x.rows <= 0) continue;
            const bool rot = x.kv == 0 && P.rs.enabled;
            // Walk every slot use in order (V tiles too), so that each wait is at most
            // one phase away from its barrier; the slot is refilled only after both
            // this release and the MMA's commit.
            for (int kb = 0; kb < P.nblk; ++kb) {
                uint32_t si = sp.idx + kb, ph = sp.phase;
                if (si >= NS) { si -= NS; ph ^= 1; }
                if (!W.wait(bar(kBarFull + si), ph)) { ok = false; break; }
            }
            if (!ok) break;
            if (!rot) {
                if (xt == 0)
                    for (int kb = 0; kb < P.nblk; ++kb) {
                        const uint32_t si = sp.idx + kb;
                        mbar_arrive(bar(kBarEmpty + (si >= NS ? si - NS : si)));
                    }
                for (int kb = 0; kb < P.nblk; ++kb) sp.adv(NS);
                continue;
            }
            const uint32_t csbuf = kc & 1;
            if (P.share_cs) {   // the epilogue must be done with this buffer's previous K tile
                if (!W.wait(bar(kBarCsFree + csbuf), ((kc >> 1) & 1) ^ 1)) break;
                tc_fence_after();
            }
            // rows past the sequence are rotated too (harmless: not stored) so that the
            // warp-collective TMEM stores below see every lane
            const int t = x.t0 + row;
            const int p = row < x.rows ? src_pos_of_seq(P.src_pos, P.src_max_seq, x.b, t, P.max_position, P.status)
                                       : 0;
#pragma unroll
            for (int cc = 0; cc < kMine; ++cc) {
                const int i = (part * kMine + cc) * 8;             // first pair index of the chunk
                float2 cs[8];
#pragma unroll
                for (int e2 = 0; e2 < 8; ++e2) cs[e2] = turn_cs(sTurnS[i + e2], p);
                if (P.share_cs) {
                    uint32_t v[16];
#pragma unroll
                    for (int e2 = 0; e2 < 8; ++e2) { v[2 * e2] = __float_as_uint(cs[e2].x); v[2 * e2 + 1] = __float_as_uint(cs[e2].y); }
                    tmem_st16(cs_lane + csbuf * (uint32_t)(2 * HS) + 2 * i, v);
                }
                for (int q = 0; q < heads; ++q) {
                    // element i (and i+HS) of head q: K-block and column within it
                    const int k_lo = q * 2 * HS + i, k_hi = k_lo + HS;
                    uint32_t s_lo = sp.idx + (k_lo >> 6), s_hi = sp.idx + (k_hi >> 6);
                    s_lo -= s_lo >= NS ? NS : 0;
                    s_hi -= s_hi >= NS ? NS : 0;
                    uint8_t* p_lo = sRing + s_lo * kBlockBytes + sw128_off(row, k_lo & 63, kTileM);
                    uint8_t* p_hi = sRing + s_hi * kBlockBytes + sw128_off(row, k_hi & 63, kTileM);
                    const uint4 wl = *reinterpret_cast<const uint4*>(p_lo);
                    const uint4 wh = *reinterpret_cast<const uint4*>(p_hi);
                    const uint32_t al[4] = {wl.x, wl.y, wl.z, wl.w};
                    const uint32_t ah[4] = {wh.x, wh.y, wh.z, wh.w};
                    uint32_t ol[4], oh[4];
#pragma unroll
                    for (int w2 = 0; w2 < 4; ++w2) {
                        float x0a = bf_lo(al[w2]), x0b = bf_hi(al[w2]);
                        float x1a = bf_lo(ah[w2]), x1b = bf_hi(ah[w2]);
                        const float2 ca = cs[2 * w2], cb = cs[2 * w2 + 1];
                        // undo the rotation: R(-theta)
                        const float u0a = fmaf(x0a, ca.x, x1a * ca.y), u1a = fmaf(x1a, ca.x, -x0a * ca.y);
                        const float u0b = fmaf(x0b, cb.x, x1b * cb.y), u1b = fmaf(x1b, cb.x, -x0b * cb.y);
                        ol[w2] = pack_bf16(u0a, u0b);
                        oh[w2] = pack_bf16(u1a, u1b);
                    }
                    *reinterpret_cast<uint4*>(p_lo) = make_uint4(ol[0], ol[1], ol[2], ol[3]);
                    *reinterpret_cast<uint4*>(p_hi) = make_uint4(oh[0], oh[1], oh[2], oh[3]);
                }
            }
            if (P.share_cs) {
                tmem_st_wait();
                tc_fence_before();
            }
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kBarKReady + kr_idx));
            if (++kr_idx == NKR) kr_idx = 0;
            ++kc;
            // the MMA's commit (after every prologue warp's "ready") completes the release
            if (xt == 0)
                for (int kb = 0; kb < P.nblk; ++kb) {
                    const uint32_t si = sp.idx + kb;
                    mbar_arrive(bar(kBarEmpty + (si >= NS ? si - NS : si)));
                }
            for (int kb = 0; kb < P.nblk; ++kb) sp.adv(NS);
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, P.tmem_cols);
    }
}

using EncodeTiled = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                 const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                 CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiled encoder()
{
    static EncodeTiled fn = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiled)p;
    }
    return fn;
}

}  // namespace

bool aligned_supported(int in_dim, int dt, int ds, int share, int Lt, int batch, int kl)
{
    // one source layer per target layer (one tensor map each) and a resident B image
    TcConfig c = tc_config(in_dim, dt, ds, share);
    return c.ok && in_dim <= 256 && kl == 1 && Lt <= KVX_MAX_ALIGNED_LAYERS && batch <= KVX_MAX_ALIGNED_BATCH &&
           encoder() != nullptr;
}

bool encode_source_map(void* map_out, const void* base, int ds, int S_max, int Hs, int batch, long long ss,
                       long long sh, long long sb)
{
    EncodeTiled enc = encoder();
    if (!enc) return false;
    const cuuint64_t dims[4] = {(cuuint64_t)ds, (cuuint64_t)(S_max > 0 ? S_max : 1), (cuuint64_t)Hs,
                                (cuuint64_t)batch};
    const cuuint64_t strides[3] = {(cuuint64_t)ss * 2, (cuuint64_t)sh * 2, (cuuint64_t)sb * 2};
    const cuuint32_t box[4] = {(cuuint32_t)kBlockK, (cuuint32_t)kTileM, 1, 1};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    return enc(reinterpret_cast<CUtensorMap*>(map_out), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base),
               dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

size_t aligned_map_bytes() { return sizeof(CUtensorMap); }

// Launch with programmatic stream serialization: the kernel may start while the
// previous kernel in the stream finishes; it waits (griddepcontrol.wait) before
// touching global memory, so stream order is preserved for every memory access.
template <typename K>
cudaError_t launch_pdl(K kernel, int grid, cudaStream_t stream, const AlignedParams& P)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemMax;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, P);
    return e != cudaSuccess ? e : cudaGetLastError();
}

template <int HS, int VAR>
static cudaError_t launch_aligned(int grid, cudaStream_t stream, const AlignedParams& P)
{
    const cudaError_t e = smem_opt_in<translate_tc_aligned_kernel<HS, VAR>>(kSmemMax);
    if (e != cudaSuccess) return e;
    return launch_pdl(translate_tc_aligned_kernel<HS, VAR>, grid, stream, P);
}

cudaError_t launch_translate_tc_aligned(const TranslateParams& T, const void* const* maps,
                                        const unsigned long long* host_turns, int num_sms, cudaStream_t stream)
{
    TcConfig cfg = tc_config(T.in_dim, T.dt, T.ds, share_heads(T));
    if (!cfg.ok || T.Lt > KVX_MAX_ALIGNED_LAYERS || T.batch > KVX_MAX_ALIGNED_BATCH) return cudaErrorNotSupported;
    static thread_local AlignedParams P;   // large (~27 KB): filled on the host, passed by value
    memset(&P, 0, offsetof(AlignedParams, maps));
    P.Hs = T.Hs; P.ds = T.ds; P.Ht = T.Ht; P.dt = T.dt; P.in_dim = T.in_dim; P.r = T.r; P.e = T.e; P.Lt = T.Lt;
    P.dense = T.dense;
    P.n_tile = cfg.n_tile;
    P.n_split = cfg.n_split;
    P.groups = T.Lt * T.Ht * 2 * cfg.n_split;
    P.nblk = T.in_dim / kBlockK;
    P.m_tiles_max = (T.T_total + kTileM - 1) / kTileM + T.batch - 1;
    P.batch = T.batch; P.src_max_seq = T.src_max_seq; P.src_seq_len = T.src_seq_len; P.src_pos = T.src_pos;
    P.T_total = T.T_total; P.seq_off = T.seq_off; P.tgt_pos = T.tgt_pos;
    P.paged = T.paged; P.dst_max_seq = T.dst_max_seq; P.db = T.db; P.dh = T.dh; P.dts = T.dts;
    P.page_table = T.page_table; P.max_pages = T.max_pages; P.page_size = T.page_size; P.num_pages = T.num_pages;
    P.rs = T.rs; P.rt = T.rt; P.max_position = T.max_position; P.status = T.status; P.w = T.w;
    P.plain_stores = T.plain_stores;
    P.wait_ns = T.wait_ns;
    P.stall_unit1 = T.stall_unit1;
    P.idesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(P.n_tile >> 3) << 17) | ((uint32_t)(kTileM >> 4) << 24);
    P.share_cs = T.rs.enabled && T.rt.enabled && T.ds == T.dt && !T.src_pos && !T.tgt_pos &&
                 T.rope_same && 2 * P.n_tile + 2 * T.dt <= 512;
    P.cs_col = (unsigned)(2 * P.n_tile);
    unsigned cols = 32;
    while (cols < 2u * (unsigned)P.n_tile + (P.share_cs ? 2u * (unsigned)T.dt : 0u)) cols <<= 1;
    P.tmem_cols = cols;
    P.b_bytes = (unsigned)(T.in_dim * P.n_tile * 2);
    P.stage_row_bytes = (unsigned)(P.n_tile * 2 + 16);
    unsigned off = 0;
    auto take = [&](unsigned bytes, unsigned align) {
        off = (off + align - 1) / align * align;
        const unsigned o = off;
        off += bytes;
        return o;
    };
    P.off_b = take(P.b_bytes, 1024);
    P.off_stage = take(kTileM * P.stage_row_bytes, 128);
    P.off_bar = take(kNumBars * 8, 8);
    P.off_misc = take(16, 16);
    P.off_seq = take((unsigned)(3 * T.batch + 2) * 4, 16);
    P.off_ring = take(0, 1024);
    // slots for a 1024-byte-aligned dynamic shared memory base (the kernel recounts for the actual
    // base); the kernel needs a full tile's K-blocks even in the worst alignment
    const int avail = kSmemMax - (int)P.off_ring;
    P.nslots = avail / kBlockBytes;
    if (P.nslots > kMaxSlots) P.nslots = kMaxSlots;
    if ((kSmemMax - 1024 - (int)P.off_ring) / kBlockBytes < P.nblk) return cudaErrorNotSupported;
    P.nkready = P.nslots / P.nblk + 2;
    for (int i = 0; i < T.ds / 2; ++i) P.turns[i] = T.rs.enabled ? host_turns[i] : 0ull;
    for (int i = 0; i < T.dt / 2; ++i) P.turns[128 + i] = T.rt.enabled ? host_turns[T.ds / 2 + i] : 0ull;
    for (int j = 0; j < T.Lt; ++j) {
        P.dst_k[j] = T.dst_k[j];
        P.dst_v[j] = T.dst_v[j];
        memcpy(&P.maps[2 * j], maps[2 * j], sizeof(CUtensorMap));
        memcpy(&P.maps[2 * j + 1], maps[2 * j + 1], sizeof(CUtensorMap));
    }
    const long long UH = (long long)(P.groups / 2) * P.m_tiles_max;
    const int grid = (int)(UH < num_sms ? UH : num_sms);
    // V shares paired with the K shares by cost (kvx_schedule.h)
    P.use_vmap = grid <= kMaxVmap;
    if (P.use_vmap) pair_v_shares(grid, UH, P.m_tiles_max, P.vmap);
    // the diagnostics' and the thread-store instantiations only when they are asked for
    const int var = P.plain_stores ? 2 : (P.wait_ns != 0 || P.stall_unit1 != 0 ? 1 : 0);
    switch (T.ds * 4 + var) {
    case 64 * 4 + 0: return launch_aligned<32, 0>(grid, stream, P);
    case 64 * 4 + 1: return launch_aligned<32, 1>(grid, stream, P);
    case 64 * 4 + 2: return launch_aligned<32, 2>(grid, stream, P);
    case 128 * 4 + 0: return launch_aligned<64, 0>(grid, stream, P);
    case 128 * 4 + 1: return launch_aligned<64, 1>(grid, stream, P);
    case 128 * 4 + 2: return launch_aligned<64, 2>(grid, stream, P);
    case 256 * 4 + 0: return launch_aligned<128, 0>(grid, stream, P);
    case 256 * 4 + 1: return launch_aligned<128, 1>(grid, stream, P);
    case 256 * 4 + 2: return launch_aligned<128, 2>(grid, stream, P);
    default: return cudaErrorNotSupported;
    }
    return cudaGetLastError();
}

}  // namespace kvx
