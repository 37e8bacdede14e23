// kvx_tc.cu -- tensor-core translation kernel for sm_103a (tcgen05 / TMEM / bulk copies).
//
// The per-(target layer, target KV head, K|V) projection of T_theta (paper
// Section 5) is a dense [T x in] . [in x d_t] contraction; everything around it
// (span gather, RoPE undo, span mean, RoPE apply, cache write) is streaming work
// fused into the GEMM's prologue and epilogue.
//
// Persistent kernel, one CTA per SM, work unit = (group, 128-token tile) with
// group = (target layer j, target head h, K|V, output split nt).  A CTA walks a
// contiguous range of units, so the group's weight tile (B operand) stays in
// shared memory across its token tiles.  Warp roles:
//   warp 0      producer: resolves the spans of each 32-token sub-tile and
//               streams the needed source rows into a byte ring in shared memory
//               with cp.async.bulk (mbarrier transaction counts); loads B images.
//   warp 1      MMA: allocates TMEM, issues tcgen05.mma (M=128, N=n_tile, K=16
//               steps over in) into a double-buffered fp32 accumulator.
//   warps 2-5   epilogue: tcgen05.ld the accumulator (one thread per token row),
//               apply the target RoPE, round to bf16, stage the row and write it
//               to the target cache (contiguous or paged) with cp.async.bulk.
//   warps 6-13  prologue: one warp per target token at a time, lanes across the
//               in channels: undo the source RoPE of each span row, take the span
//               mean, round to bf16 and store the A tile in the UMMA K-major
//               128-byte-swizzled layout.
// Every wait is a bounded mbarrier poll: after ~1 s it records
// KVX_DEV_WAIT_TIMEOUT, raises a CTA-wide abort flag and the kernel drains and
// returns (no trap, no hang).
#include "kvx_common.cuh"
#include "kvx_kernels.h"
#include "kvx_tc_common.cuh"

namespace kvx {
namespace {

constexpr int kTileM = 128;
constexpr int kSub = 32;
constexpr int kSubPerTile = kTileM / kSub;
constexpr int kNumSlots = 8;
constexpr int kProducerWarp = 0;
constexpr int kMmaWarp = 1;
constexpr int kEpiWarp0 = 2;
constexpr int kNumEpiWarps = 8;               // two per TMEM lane quadrant, splitting the rotary pairs
constexpr int kXfWarp0 = kEpiWarp0 + kNumEpiWarps;
constexpr int kNumXfWarps = 8;
constexpr int kThreads = (kXfWarp0 + kNumXfWarps) * 32;
constexpr int kMaxSeqCache = 512;         // sequences whose metadata is kept in shared memory

// barrier indices
constexpr int kBarBFull = 0, kBarBEmpty = 1, kBarAFull = 2, kBarAEmpty = 3;
constexpr int kBarDFull = 4;               // +buf (2)
constexpr int kBarDEmpty = 6;              // +buf (2)
constexpr int kBarSlotFull = 8;            // +slot
constexpr int kBarSlotEmpty = 8 + kNumSlots;
constexpr int kBarPair = 8 + 2 * kNumSlots;   // +quad*2+{0,1}: the two epilogue warps of a quadrant meet
constexpr int kNumBars = kBarPair + 8;

struct SubMeta {
    int stage_row;   // stage row of the span start; < 0: rows are read from global memory
    int lo, hi;      // source span within the sequence (hi <= lo: nothing to gather)
    int b;           // sequence
};

struct SlotHdr {
    unsigned rows;     // rows per head staged for the sub-tile
    unsigned offset;   // byte offset of the sub-tile's region in the ring
};

struct TcLaunch {
    int n_tile, n_split, in_dim, groups, m_tiles;
    unsigned b_bytes, a_bytes, row_bytes, stage_row_bytes, ring_bytes;
    unsigned off_b, off_a, off_stage, off_ring, off_meta, off_hdr, off_bar, off_misc, off_seq, off_turns, off_slot;
    int seq_cached;   // per-sequence offsets and source lengths copied to shared memory
    unsigned idesc;
    unsigned tmem_cols;
};

struct Unit {
    int j, h, kv, nt, tile, g;
};
__device__ __forceinline__ Unit make_unit(int g, int tile, const TcLaunch& L, int Ht)
{
    Unit x;
    x.g = g;
    x.tile = tile;
    int rest = g;
    x.nt = rest % L.n_split;
    rest /= L.n_split;
    x.kv = rest & 1;
    rest >>= 1;
    x.h = rest % Ht;
    x.j = rest / Ht;
    return x;
}
// The CTA's units: an equal share of the K units, then of the V units (each share
// group-major, so a group's weights stay resident), walked with counters only.
struct Walker {
    int count, nK, it;
    int kv, j, h, nt, tile;
    int u0, v0, m_tiles, n_split, Ht;
    Unit x;
    __device__ __forceinline__ void fill()
    {
        x.j = j; x.h = h; x.kv = kv; x.nt = nt; x.tile = tile;
        x.g = ((j * Ht + h) * 2 + kv) * n_split + nt;
    }
    __device__ __forceinline__ void seek(int idx, int kv_)
    {
        kv = kv_;
        const int hg = idx / m_tiles;
        tile = idx - hg * m_tiles;
        nt = hg % n_split;
        const int jh = hg / n_split;
        h = jh % Ht;
        j = jh / Ht;
        fill();
    }
    __device__ __forceinline__ void start(const TcLaunch& L, int Ht_)
    {
        m_tiles = L.m_tiles; n_split = L.n_split; Ht = Ht_;
        const long long UH = (long long)(L.groups / 2) * L.m_tiles;
        const int G = gridDim.x, c = blockIdx.x, vr = G - 1 - c;
        u0 = (int)((long long)c * UH / G);
        const int u1 = (int)((long long)(c + 1) * UH / G);
        v0 = (int)((long long)vr * UH / G);
        const int v1 = (int)((long long)(vr + 1) * UH / G);
        nK = u1 - u0;
        count = nK + (v1 - v0);
        it = 0;
        if (nK > 0) seek(u0, 0);
        else if (count > 0) seek(v0, 1);
    }
    __device__ __forceinline__ bool more() const { return it < count; }
    __device__ __forceinline__ void next()
    {
        if (++it >= count) return;
        if (it == nK) { seek(v0, 1); return; }
        if (++tile == m_tiles) {
            tile = 0;
            if (++nt == n_split) {
                nt = 0;
                if (++h == Ht) { h = 0; ++j; }
            }
        }
        fill();
    }
    __device__ __forceinline__ bool last_of_group() const
    {
        return it + 1 == count || it + 1 == nK || tile + 1 == m_tiles;
    }
};

// Sequence metadata view: shared-memory copies of seq_off / src_seq_len when the
// batch is small enough, else the global arrays.
struct SeqView {
    const int* off;    // [batch+1]
    const int* slen;   // [batch]
    int batch;
    __device__ __forceinline__ int find(int tp) const
    {
        int lo = 0, hi = batch - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (off[mid] <= tp) lo = mid; else hi = mid - 1;
        }
        return lo;
    }
};

// Source-side resolution of one target token (sequence, clamped span).
__device__ __forceinline__ void resolve_src(const TranslateParams& P, const SeqView& sv, int tp, int& b, int& lo,
                                            int& hi)
{
    b = sv.find(tp);
    const int t = tp - sv.off[b];
    int S = sv.slen[b];
    if (S > P.src_max_seq || S < 0) {
        set_status(P.status, KVX_DEV_SEQ_CLAMPED);
        S = S < 0 ? 0 : P.src_max_seq;
    }
    if (P.span_lo) { lo = __ldg(&P.span_lo[tp]); hi = __ldg(&P.span_hi[tp]); }
    else { lo = t; hi = t + 1; }
    if (lo < 0 || hi > S || hi <= lo) {
        set_status(P.status, KVX_DEV_SPAN_CLAMPED);
        lo = lo < 0 ? 0 : (lo > S - 1 ? S - 1 : lo);
        hi = hi > S ? S : hi;
        if (hi <= lo) hi = lo + 1;
        if (S == 0) { lo = 0; hi = 0; }
    }
}

// Target-side resolution: output row offset (-1: not written) and RoPE position.
__device__ __forceinline__ void resolve_dst(const TranslateParams& P, const SeqView& sv, int tp, long long& dst_off,
                                            int& pt)
{
    const int b = sv.find(tp);
    const int t = tp - sv.off[b];
    const int p = P.tgt_pos ? __ldg(&P.tgt_pos[tp]) : t;
    pt = P.rt.enabled ? clamp_pos(p, P.max_position, P.status) : 0;
    if (!P.paged) {
        if (t >= P.dst_max_seq) { set_status(P.status, KVX_DEV_SEQ_CLAMPED); dst_off = -1; }
        else dst_off = (long long)b * P.db + (long long)t * P.dts;
    } else {
        const int pi = t / P.page_size;
        const int page = pi < P.max_pages ? __ldg(&P.page_table[(size_t)b * P.max_pages + pi]) : -1;
        if (page < 0 || page >= P.num_pages) { set_status(P.status, KVX_DEV_PAGE_INVALID); dst_off = -1; }
        else dst_off = ((long long)page * P.page_size + (t % P.page_size)) * (long long)P.Ht * P.dt;
    }
}

// (cos, sin) for PP consecutive frequencies i0.. at position p, from the
// fixed-point turns held in shared memory.
template <int PP>
__device__ __forceinline__ void rope_cs_vec(const unsigned long long* turns, int p, int i0, float2 (&cs)[PP])
{
#pragma unroll
    for (int q = 0; q < PP; ++q) cs[q] = turn_cs(turns[i0 + q], p);
}

// ------------------------------------------------------------------ the kernel
template <int PP>
__global__ void __launch_bounds__(kThreads, 1)
translate_tc_kernel(const __grid_constant__ TranslateParams P, const __grid_constant__ TcLaunch L)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* sB = smem + L.off_b;
    uint8_t* sA = smem + L.off_a;
    uint8_t* sStage = smem + L.off_stage;
    uint8_t* sRing = smem + L.off_ring;
    SubMeta* sMeta = reinterpret_cast<SubMeta*>(smem + L.off_meta);
    SlotHdr* sHdr = reinterpret_cast<SlotHdr*>(smem + L.off_hdr);
    uint64_t* sBar = reinterpret_cast<uint64_t*>(smem + L.off_bar);
    volatile int* sAbort = reinterpret_cast<volatile int*>(smem + L.off_misc);
    uint32_t* sTmemBase = reinterpret_cast<uint32_t*>(smem + L.off_misc + 4);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    auto bar = [&](int i) { return smem_u32(&sBar[i]); };

    if (threadIdx.x == 0) {
        *sAbort = 0;
        mbar_init(bar(kBarBFull), 1);
        mbar_init(bar(kBarBEmpty), 1);
        mbar_init(bar(kBarAFull), kNumXfWarps);
        mbar_init(bar(kBarAEmpty), 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar(kBarDFull + i), 1);
            mbar_init(bar(kBarDEmpty + i), kNumEpiWarps);
        }
        for (int i = 0; i < kNumSlots; ++i) {
            mbar_init(bar(kBarSlotFull + i), 1);
            mbar_init(bar(kBarSlotEmpty + i), kNumXfWarps);
        }
        for (int i = 0; i < 8; ++i) mbar_init(bar(kBarPair + i), 2);
        fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        tmem_alloc(smem_u32(sTmemBase), L.tmem_cols);
        tmem_relinquish();
    }
    // Nothing above touched global memory: with programmatic dependent launch that set-up
    // overlaps the previous kernel in the stream; everything below waits for it.
    grid_dependency_wait();
    grid_launch_dependents();
    unsigned long long* sTurnS = reinterpret_cast<unsigned long long*>(smem + L.off_turns);
    unsigned long long* sTurnT = sTurnS + (P.ds >> 1);
    for (int i = threadIdx.x; i < (P.ds >> 1); i += blockDim.x) sTurnS[i] = P.rs.enabled ? __ldg(&P.rs.turns[i]) : 0ull;
    for (int i = threadIdx.x; i < (P.dt >> 1); i += blockDim.x) sTurnT[i] = P.rt.enabled ? __ldg(&P.rt.turns[i]) : 0ull;
    int* sSeqOff = reinterpret_cast<int*>(smem + L.off_seq);
    int* sSrcLen = sSeqOff + kMaxSeqCache + 1;
    if (L.seq_cached) {
        for (int i = threadIdx.x; i <= P.batch; i += blockDim.x) sSeqOff[i] = __ldg(&P.seq_off[i]);
        for (int i = threadIdx.x; i < P.batch; i += blockDim.x) sSrcLen[i] = __ldg(&P.src_seq_len[i]);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *sTmemBase;

    const Waiter W{sAbort, P.status};
    const SeqView sv{L.seq_cached ? sSeqOff : P.seq_off, L.seq_cached ? sSrcLen : P.src_seq_len, P.batch};

    const int hw = L.n_tile >> 1;                 // pair half-width of an output split
    const int half_t = P.dt >> 1;

    if (warp == kProducerWarp) {
        // ------------------------------------------------------------ producer
        const uint64_t pol_stream = policy_evict_first();
        const uint64_t pol_keep = policy_evict_last();
        const int r_heads = L.in_dim / P.ds;         // source heads per A row (1 when expanding)
        const bool rows_contig = P.ss == P.ds;
        int cur_g = -1;
        uint32_t b_loads = 0, issued = 0, released = 0;
        unsigned long long head = 0;                 // monotonic ring byte counter
        unsigned long long* slot_start = reinterpret_cast<unsigned long long*>(smem + L.off_slot);   // lane 0's copy
        bool ok = true;
        // wait until sub-tile k (0-based) has been released by the prologue warps
        auto release_upto = [&](uint32_t k) -> bool {
            while (released < k) {
                if (!W.wait(bar(kBarSlotEmpty + released % kNumSlots), (released / kNumSlots) & 1)) return false;
                ++released;
            }
            return true;
        };
        Walker wk;
        for (wk.start(L, P.Ht); wk.more() && ok; wk.next()) {
            const Unit& x = wk.x;
            if (x.g != cur_g) {
                if (!W.wait(bar(kBarBEmpty), (b_loads & 1) ^ 1)) { ok = false; break; }
                if (lane == 0) mbar_arrive_expect_tx(bar(kBarBFull), L.b_bytes);
                __syncwarp();
                const uint8_t* img = (const uint8_t*)P.w + (size_t)x.g * L.b_bytes;
                const uint32_t piece = L.b_bytes / 4;
                if (lane < 4)
                    bulk_g2s(smem_u32(sB) + lane * piece, img + (size_t)lane * piece, piece, bar(kBarBFull), pol_keep);
                ++b_loads;
                cur_g = x.g;
            }
            const __nv_bfloat16* src = (const __nv_bfloat16*)(x.kv ? P.src_v[x.j] : P.src_k[x.j]);
            const int g0 = P.r > 1 ? x.h * P.r : x.h / P.e;
            // spans of the tile's 128 tokens, 4 per lane, loads issued together
            int rb[kSubPerTile], rlo[kSubPerTile], rhi[kSubPerTile];
#pragma unroll
            for (int sq = 0; sq < kSubPerTile; ++sq) {
                const int tp = x.tile * kTileM + sq * kSub + lane;
                rb[sq] = -1; rlo[sq] = 0; rhi[sq] = 0;
                if (tp < P.T_total) resolve_src(P, sv, tp, rb[sq], rlo[sq], rhi[sq]);
            }
#pragma unroll 1
            for (int sq = 0; sq < kSubPerTile; ++sq) {
                const int tp = x.tile * kTileM + sq * kSub + lane;
                const bool valid = tp < P.T_total;
                int b = rb[0], lo = rlo[0], hi = rhi[0];
#pragma unroll
                for (int z = 1; z < kSubPerTile; ++z)
                    if (sq == z) { b = rb[z]; lo = rlo[z]; hi = rhi[z]; }
                const int b_prev = __shfl_up_sync(0xffffffffu, b, 1);
                const int lo_prev = __shfl_up_sync(0xffffffffu, lo, 1);
                const int hi_prev = __shfl_up_sync(0xffffffffu, hi, 1);
                const bool first = valid && (lane == 0 || b_prev != b);
                const bool nonmono = valid && !first && (lo < lo_prev || hi < hi_prev);
                const int cover = first ? lo : max(lo, hi_prev);
                const int n_new = valid ? max(0, hi - cover) : 0;
                int incl = n_new;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int v = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += v;
                }
                const int start = incl - n_new;
                const unsigned R = (unsigned)__shfl_sync(0xffffffffu, incl, 31);
                const unsigned need_rows = R * (unsigned)r_heads;
                const bool direct = __any_sync(0xffffffffu, nonmono) ||
                                    (unsigned long long)need_rows * L.row_bytes + 128ull * r_heads > L.ring_bytes;
                const unsigned hstride = R * L.row_bytes + 128;   // pad: the head halves of a warp hit different banks
                const unsigned need = direct || R == 0 ? 0u : (unsigned)r_heads * hstride;

                // slot reuse and ring space
                const uint32_t slot = issued % kNumSlots;
                if (issued >= kNumSlots && !release_upto(issued - kNumSlots + 1)) { ok = false; break; }
                unsigned long long off = head;
                if (need) {
                    if (off % L.ring_bytes + need > L.ring_bytes) off = (off / L.ring_bytes + 1) * L.ring_bytes;
                    while (true) {
                        const unsigned long long tail = released == issued ? off : slot_start[released % kNumSlots];
                        if (off + need - tail <= L.ring_bytes) break;
                        if (!release_upto(released + 1)) { ok = false; break; }
                    }
                    if (!ok) break;
                }
                head = off + need;
                slot_start[slot] = off;
                const unsigned roff = (unsigned)(off % L.ring_bytes);

                SubMeta mt;
                mt.stage_row = direct ? -1 : start - (cover - lo);
                mt.lo = lo;
                mt.hi = hi;
                mt.b = b;
                if (!valid) { mt.lo = 0; mt.hi = 0; mt.b = 0; }
                sMeta[slot * kSub + lane] = mt;
                if (lane == 0) sHdr[slot] = SlotHdr{R, roff};
                __threadfence_block();
                __syncwarp();
                if (lane == 0) {
                    if (need) mbar_arrive_expect_tx(bar(kBarSlotFull + slot), need_rows * L.row_bytes);   // bytes copied
                    else mbar_arrive(bar(kBarSlotFull + slot));
                }
                __syncwarp();
                if (need) {
                    const uint32_t ring0 = smem_u32(sRing) + roff;
                    if (rows_contig) {
                        // one copy per (contiguous run of source rows, head)
                        const bool run_start = n_new > 0 && (first || lo > hi_prev);
                        const unsigned runs = __ballot_sync(0xffffffffu, run_start);
                        const unsigned later = lane < 31 ? runs & (0xffffffffu << (lane + 1)) : 0u;
                        const int nxt = later ? __ffs(later) - 1 : 32;
                        const int nxt_start = __shfl_sync(0xffffffffu, start, nxt < 32 ? nxt : lane);
                        if (run_start) {
                            const unsigned rows = (nxt < 32 ? (unsigned)nxt_start : R) - (unsigned)start;
                            for (int q = 0; q < r_heads; ++q) {
                                const __nv_bfloat16* s0 =
                                    src + (long long)b * P.sb + (long long)(g0 + q) * P.sh + (long long)cover * P.ss;
                                bulk_g2s(ring0 + (unsigned)q * hstride + (unsigned)start * L.row_bytes, s0,
                                         rows * L.row_bytes, bar(kBarSlotFull + slot), pol_stream);
                            }
                        }
                    } else {
                        for (int s = cover; s < cover + n_new; ++s)
                            for (int q = 0; q < r_heads; ++q) {
                                const __nv_bfloat16* s0 =
                                    src + (long long)b * P.sb + (long long)(g0 + q) * P.sh + (long long)s * P.ss;
                                bulk_g2s(ring0 + (unsigned)q * hstride + (unsigned)(start + s - cover) * L.row_bytes,
                                         s0, L.row_bytes, bar(kBarSlotFull + slot), pol_stream);
                            }
                    }
                }
                ++issued;
            }
        }
        // on abort, let copies already in flight land before the CTA leaves
        if (*sAbort) {
            const unsigned long long t0 = globaltimer();
            for (uint32_t c = issued > kNumSlots ? issued - kNumSlots : 0; c < issued; ++c)
                while (!mbar_try_wait(bar(kBarSlotFull + c % kNumSlots), (c / kNumSlots) & 1) &&
                       globaltimer() - t0 < kWaitNs) {}
            if (b_loads)
                while (!mbar_try_wait(bar(kBarBFull), (b_loads - 1) & 1) && globaltimer() - t0 < kWaitNs) {}
        }
    } else if (warp == kMmaWarp) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            int cur_g = -1;
            uint32_t b_cnt = 0, tcount = 0;
            Walker wk;
            for (wk.start(L, P.Ht); wk.more(); wk.next()) {
                const Unit& x = wk.x;
                if (x.g != cur_g) {
                    if (!W.wait(bar(kBarBFull), b_cnt & 1)) break;
                    ++b_cnt;
                    cur_g = x.g;
                }
                const uint32_t buf = tcount & 1;
                if (!W.wait(bar(kBarDEmpty + buf), ((tcount >> 1) & 1) ^ 1)) break;
                if (!W.wait(bar(kBarAFull), tcount & 1)) break;
                tc_fence_after();
                const uint32_t d = tmem_base + buf * (uint32_t)L.n_tile;
                const uint32_t a0 = smem_u32(sA), b0 = smem_u32(sB);
                for (int kk = 0; kk < L.in_dim / 16; ++kk) {
                    const uint32_t kb = kk >> 2, ko = (kk & 3) * 32;
                    const uint64_t ad = sw128_desc(a0 + kb * (kTileM * 128) + ko);
                    const uint64_t bd = sw128_desc(b0 + kb * (L.n_tile * 128) + ko);
                    umma_bf16(d, ad, bd, L.idesc, kk > 0 ? 1u : 0u);
                }
                umma_commit(bar(kBarAEmpty));
                umma_commit(bar(kBarDFull + buf));
                const bool last_of_group = wk.last_of_group();
                if (last_of_group) umma_commit(bar(kBarBEmpty));
                ++tcount;
            }
        }
        __syncwarp();
    } else if (warp < kEpiWarp0 + kNumEpiWarps) {
        // ------------------------------------------------------------ epilogue
        const int quad = warp & 3;
        const int half = (warp - kEpiWarp0) >> 2;          // which half of the rotary pairs
        const int m = quad * 32 + lane;
        const int pc_begin = half * (hw >> 1), pc_end = pc_begin + (hw >> 1);
        uint8_t* srow = sStage + (size_t)m * L.stage_row_bytes;
        const uint32_t srow_u32 = smem_u32(srow);
        uint32_t tcount = 0;
        Walker wk;
        for (wk.start(L, P.Ht); wk.more(); wk.next()) {
            const Unit& x = wk.x;
            const uint32_t buf = tcount & 1;
            // resolve the output row while the tile is still being computed
            const int tp = x.tile * kTileM + m;
            const bool valid = tp < P.T_total;
            long long dst_off = -1;
            int pt = 0;
            if (valid) resolve_dst(P, sv, tp, dst_off, pt);
            const bool rot = x.kv == 0 && P.rt.enabled;
            float2 cs[8];
            if (rot) rope_cs_vec<8>(sTurnT, pt, x.nt * hw + pc_begin, cs);
            if (!W.wait(bar(kBarDFull + buf), (tcount >> 1) & 1)) break;
            tc_fence_after();
            // the staging row is shared by the two warps of this quadrant; the row's
            // previous store (issued by the half-0 thread) must have read it
            if (half == 0) bulk_wait_read0();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kBarPair + quad * 2));
            if (!W.wait(bar(kBarPair + quad * 2), tcount & 1)) break;
            const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + buf * (uint32_t)L.n_tile;
            for (int pc = pc_begin; pc < pc_end; pc += 8) {
                float2 csn[8];
                if (rot && pc + 8 < pc_end) rope_cs_vec<8>(sTurnT, pt, x.nt * hw + pc + 8, csn);
                uint32_t r0[8], r1[8];
                tmem_ld8(taddr + pc, r0);
                tmem_ld8(taddr + hw + pc, r1);
                tmem_ld_wait();
                float y0[8], y1[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) { y0[e] = __uint_as_float(r0[e]); y1[e] = __uint_as_float(r1[e]); }
                if (rot) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const float a = y0[e], bb = y1[e];
                        y0[e] = fmaf(a, cs[e].x, -bb * cs[e].y);
                        y1[e] = fmaf(bb, cs[e].x, a * cs[e].y);
                    }
#pragma unroll
                    for (int e = 0; e < 8; ++e) cs[e] = csn[e];
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
            if (lane == 0) mbar_arrive(bar(kBarDEmpty + buf));
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kBarPair + quad * 2 + 1));
            if (!W.wait(bar(kBarPair + quad * 2 + 1), tcount & 1)) break;
            if (half == 0 && valid && dst_off >= 0) {
                __nv_bfloat16* dst = (__nv_bfloat16*)(x.kv ? P.dst_v[x.j] : P.dst_k[x.j]) + dst_off +
                                     dst_head_off(P, x.h);
                if (L.n_split == 1) {
                    bulk_s2g(dst, srow_u32, (uint32_t)P.dt * 2);
                } else {
                    bulk_s2g(dst + x.nt * hw, srow_u32, (uint32_t)hw * 2);
                    bulk_s2g(dst + half_t + x.nt * hw, srow_u32 + hw * 2, (uint32_t)hw * 2);
                }
                bulk_commit();
            }
            ++tcount;
        }
        bulk_wait0();
    } else {
        // ------------------------------------------------------------ prologue (A tile)
        const int tw = warp - kXfWarp0;
        const int lanes_per_head = 32 * P.ds / L.in_dim;
        const int q = lane / lanes_per_head;              // head within the A row
        const int i0 = (lane % lanes_per_head) * PP;      // first rotary pair of this lane
        const int hs = P.ds >> 1;
        const int k0 = q * P.ds + i0, k1 = k0 + hs;       // A columns of the two halves
        // Two heads per A row: the lanes of head 0 and head 1 rotate the same
        // frequencies at the same positions, so each computes half and they swap.
        const bool share = lanes_per_head == 16 && PP >= 2;
        constexpr int kHalf = PP >= 2 ? PP / 2 : 1;
        unsigned long long turn[PP];
#pragma unroll
        for (int e = 0; e < PP; ++e) {
            const int f = share ? i0 + (q * kHalf + e) % PP : i0 + e;   // share: first kHalf entries are own
            turn[e] = sTurnS[f];
        }
        uint32_t sub = 0, tcount = 0;
        bool ok = true;
        Walker wk;
        for (wk.start(L, P.Ht); wk.more() && ok; wk.next()) {
            const Unit& x = wk.x;
            const bool rot = x.kv == 0 && P.rs.enabled;
            const __nv_bfloat16* src = (const __nv_bfloat16*)(x.kv ? P.src_v[x.j] : P.src_k[x.j]);
            const int g = (P.r > 1 ? x.h * P.r : x.h / P.e) + q;
            if (!W.wait(bar(kBarAEmpty), (tcount & 1) ^ 1)) break;
            for (int sq = 0; sq < kSubPerTile; ++sq) {
                const uint32_t slot = sub % kNumSlots;
                if (!W.wait(bar(kBarSlotFull + slot), (sub / kNumSlots) & 1)) { ok = false; break; }
                const SlotHdr hdr = sHdr[slot];
                // heads of a staged sub-tile are 128 bytes off bank alignment (see producer)
                const uint8_t* ring = sRing + hdr.offset + q * (hdr.rows * L.row_bytes + 128);
                // the warp's tokens of the sub-tile, kTok at a time (fewer when rows are wide,
                // to stay within the register budget)
                constexpr int kTok = PP == 4 ? 2 : kSub / kNumXfWarps;
                for (int tg = 0; tg < kSub / kNumXfWarps; tg += kTok) {
                SubMeta mt[kTok];
                int n[kTok];
                int maxn = 0;
                bool copy_only = !rot;
#pragma unroll
                for (int u4 = 0; u4 < kTok; ++u4) {
                    const int tt = tw + (tg + u4) * kNumXfWarps;
                    mt[u4] = sMeta[slot * kSub + tt];
                    const bool valid = x.tile * kTileM + sq * kSub + tt < P.T_total;
                    n[u4] = valid ? max(mt[u4].hi - mt[u4].lo, 0) : -1;
                    maxn = max(maxn, n[u4]);
                    copy_only = copy_only && n[u4] <= 1 && mt[u4].stage_row >= 0;
                }
                if (copy_only) {
                    // V rows with single-token spans: the A row is the source row itself
#pragma unroll
                    for (int u4 = 0; u4 < kTok; ++u4) {
                        const int row = sq * kSub + tw + (tg + u4) * kNumXfWarps;
                        if (n[u4] < 0) continue;
                        typename Raw<PP>::T w0, w1;
                        if (n[u4] == 1) {
                            const __nv_bfloat16* rp =
                                reinterpret_cast<const __nv_bfloat16*>(ring + (size_t)mt[u4].stage_row * L.row_bytes);
                            w0 = load_raw<PP>(rp + i0);
                            w1 = load_raw<PP>(rp + hs + i0);
                        } else {
                            w0 = typename Raw<PP>::T{};
                            w1 = typename Raw<PP>::T{};
                        }
                        *reinterpret_cast<typename Raw<PP>::T*>(sA + sw128_off(row, k0, kTileM)) = w0;
                        *reinterpret_cast<typename Raw<PP>::T*>(sA + sw128_off(row, k1, kTileM)) = w1;
                    }
                } else {
                    float a0[kTok][PP], a1[kTok][PP];
#pragma unroll
                    for (int u4 = 0; u4 < kTok; ++u4)
#pragma unroll
                        for (int e = 0; e < PP; ++e) { a0[u4][e] = 0.f; a1[u4][e] = 0.f; }
                    for (int o = 0; o < maxn; ++o) {
                        typename Raw<PP>::T w0[kTok], w1[kTok];
#pragma unroll
                        for (int u4 = 0; u4 < kTok; ++u4) {
                            if (o < n[u4]) {
                                const int srow = mt[u4].lo + o;
                                const __nv_bfloat16* rp;
                                if (mt[u4].stage_row >= 0)
                                    rp = reinterpret_cast<const __nv_bfloat16*>(
                                        ring + (size_t)(mt[u4].stage_row + o) * L.row_bytes);
                                else
                                    rp = src + (long long)mt[u4].b * P.sb + (long long)g * P.sh +
                                         (long long)srow * P.ss;
                                w0[u4] = load_raw<PP>(rp + i0);
                                w1[u4] = load_raw<PP>(rp + hs + i0);
                            }
                        }
#pragma unroll
                        for (int u4 = 0; u4 < kTok; ++u4) {
                            // rows beyond a token's span leave its sums untouched; the sine/cosine
                            // exchange below is warp-wide, so every lane takes part
                            const bool act = o < n[u4];
                            float x0[PP], x1[PP];
                            unpack(w0[u4], x0);
                            unpack(w1[u4], x1);
                            if (rot) {
                                const int pos = act ? src_pos_of(P, mt[u4].b, mt[u4].lo + o) : 0;
                                float2 cs[PP];
                                if (share) {
#pragma unroll
                                    for (int e = 0; e < kHalf; ++e) cs[e] = turn_cs(turn[e], pos);
#pragma unroll
                                    for (int e = 0; e < kHalf; ++e) {
                                        cs[kHalf + e].x = __shfl_xor_sync(0xffffffffu, cs[e].x, 16);
                                        cs[kHalf + e].y = __shfl_xor_sync(0xffffffffu, cs[e].y, 16);
                                    }
                                    if (q) {   // own entries are the second half of the lane's pairs
#pragma unroll
                                        for (int e = 0; e < kHalf; ++e) {
                                            const float2 t = cs[e];
                                            cs[e] = cs[kHalf + e];
                                            cs[kHalf + e] = t;
                                        }
                                    }
                                } else {
#pragma unroll
                                    for (int e = 0; e < PP; ++e) cs[e] = turn_cs(turn[e], pos);
                                }
#pragma unroll
                                for (int e = 0; e < PP; ++e) {
                                    // undo the rotation: R(-theta)
                                    const float u0 = fmaf(x0[e], cs[e].x, x1[e] * cs[e].y);
                                    const float u1 = fmaf(x1[e], cs[e].x, -x0[e] * cs[e].y);
                                    x0[e] = u0;
                                    x1[e] = u1;
                                }
                            }
                            if (act) {
#pragma unroll
                                for (int e = 0; e < PP; ++e) { a0[u4][e] += x0[e]; a1[u4][e] += x1[e]; }
                            }
                        }
                    }
#pragma unroll
                    for (int u4 = 0; u4 < kTok; ++u4) {
                        if (n[u4] < 0) continue;
                        const int row = sq * kSub + tw + (tg + u4) * kNumXfWarps;
                        // span mean; 1/n is exact for n = 1, 2 (the common spans)
                        const float inv_n = n[u4] > 0 ? __frcp_rn((float)n[u4]) : 0.f;
#pragma unroll
                        for (int e = 0; e < PP; ++e) {
                            a0[u4][e] *= inv_n;
                            a1[u4][e] *= inv_n;
                        }
                        store_bf16_smem<PP>(sA + sw128_off(row, k0, kTileM), a0[u4]);
                        store_bf16_smem<PP>(sA + sw128_off(row, k1, kTileM), a1[u4]);
                    }
                }
                }   // token groups
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(kBarSlotEmpty + slot));
                ++sub;
            }
            if (!ok) break;
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar(kBarAFull));
            ++tcount;
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, L.tmem_cols);
    }
}

// Weight images: for group g = ((j*Ht + h)*2 + kv)*n_split + nt, the B operand
// [n_tile rows = output columns][in] in K-major SW128 layout.  Output column of
// image row n: n < n_tile/2 -> nt*hw + n, else d_t/2 + nt*hw + (n - hw), so an
// image holds whole RoPE pairs.
__global__ void tc_weight_relayout_kernel(const __nv_bfloat16* __restrict__ wk, const __nv_bfloat16* __restrict__ wv,
                                          uint8_t* __restrict__ img, int Lt, int Ht, int in_dim, int dt, int n_tile)
{
    const int n_split = dt / n_tile, hw = n_tile / 2;
    const long long chunks_per_img = (long long)n_tile * in_dim / 8;
    const long long total = (long long)Lt * Ht * 2 * n_split * chunks_per_img;
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= total) return;
    const int gimg = (int)(idx / chunks_per_img);
    const int c = (int)(idx - (long long)gimg * chunks_per_img);   // chunk within image
    int rest = gimg;
    const int nt = rest % n_split; rest /= n_split;
    const int kv = rest & 1; rest >>= 1;
    const int h = rest % Ht;
    const int j = rest / Ht;
    // chunk c enumerates (n, k/8) with k fastest
    const int n = c / (in_dim / 8);
    const int k8 = c - n * (in_dim / 8);
    const int col = n < hw ? nt * hw + n : dt / 2 + nt * hw + (n - hw);
    const __nv_bfloat16* w = (kv ? wv : wk) + ((size_t)j * Ht + h) * (size_t)in_dim * dt;
    uint32_t v[4];
    for (int e = 0; e < 4; ++e) {
        const int k = k8 * 8 + 2 * e;
        const __nv_bfloat16 lo = w[(size_t)k * dt + col];
        const __nv_bfloat16 hi = w[(size_t)(k + 1) * dt + col];
        v[e] = (uint32_t)__bfloat16_as_ushort(lo) | ((uint32_t)__bfloat16_as_ushort(hi) << 16);
    }
    const int k = k8 * 8;
    const size_t off = (size_t)gimg * ((size_t)n_tile * in_dim * 2) + (size_t)(k >> 6) * n_tile * 128 +
                       (size_t)(n >> 3) * 1024 + (n & 7) * 128 + ((((k >> 3) & 7) ^ (n & 7)) << 4);
    *reinterpret_cast<uint4*>(img + off) = make_uint4(v[0], v[1], v[2], v[3]);
}

uint32_t make_idesc(int M, int N)
{
    return (1u << 4)                  // D format: f32
           | (1u << 7)                // A format: bf16
           | (1u << 10)               // B format: bf16
           | ((uint32_t)(N >> 3) << 17)
           | ((uint32_t)(M >> 4) << 24);   // A and B K-major, no negate, dense
}

bool tc_layout(int in_dim, int dt, int ds, TcLaunch& L)
{
    if (in_dim % 64 || in_dim > 256 || in_dim < 64) return false;
    if (dt != 64 && dt != 128 && dt != 256) return false;
    if (ds != 64 && ds != 128 && ds != 256) return false;
    if (in_dim % ds) return false;
    L.in_dim = in_dim;
    L.n_tile = (in_dim * dt * 2 <= 65536) ? dt : dt / 2;
    L.n_split = dt / L.n_tile;
    L.b_bytes = (unsigned)(in_dim * L.n_tile * 2);
    L.a_bytes = (unsigned)(kTileM * in_dim * 2);
    L.row_bytes = (unsigned)(ds * 2);
    L.stage_row_bytes = (unsigned)(L.n_tile * 2 + 16);
    unsigned off = 0;
    auto take = [&](unsigned bytes, unsigned align) {
        off = (off + align - 1) / align * align;
        const unsigned o = off;
        off += bytes;
        return o;
    };
    L.off_b = take(L.b_bytes, 1024);
    L.off_a = take(L.a_bytes, 1024);
    L.off_stage = take(kTileM * L.stage_row_bytes, 128);
    L.off_meta = take(kNumSlots * kSub * sizeof(SubMeta), 16);
    L.off_hdr = take(kNumSlots * sizeof(SlotHdr), 16);
    L.off_bar = take(kNumBars * 8, 8);
    L.off_misc = take(16, 16);
    L.off_seq = take((2 * kMaxSeqCache + 1) * sizeof(int), 16);
    L.off_turns = take((unsigned)(ds / 2 + dt / 2) * 8, 16);
    L.off_slot = take(kNumSlots * 8, 16);
    L.off_ring = (off + 127) / 128 * 128;
    const int avail = kSmemMax - 1024 - (int)L.off_ring;   // 1024: alignment slack of the dynamic base
    L.ring_bytes = avail > 0 ? (unsigned)(avail / 1024 * 1024) : 0;
    if (L.ring_bytes < (3u * kSub * L.row_bytes + 128u) * (unsigned)(in_dim / ds)) return false;   // one worst sub-tile
    L.idesc = make_idesc(kTileM, L.n_tile);
    unsigned cols = 32;
    while (cols < 2u * (unsigned)L.n_tile) cols <<= 1;
    L.tmem_cols = cols;
    return cols <= 512;
}

}  // namespace

TcConfig tc_config(int in_dim, int dt, int ds)
{
    TcLaunch L{};
    TcConfig c{0, 0, 0, kThreads, 0};
    if (!tc_layout(in_dim, dt, ds, L)) return c;
    c.n_tile = L.n_tile;
    c.n_split = L.n_split;
    c.smem_bytes = kSmemMax;
    c.ok = 1;
    return c;
}

size_t tc_weight_image_bytes(int in_dim, int dt, int Lt, int Ht)
{
    return (size_t)Lt * Ht * 2 * (size_t)in_dim * dt * 2;
}

cudaError_t launch_tc_weight_relayout(const void* w_k, const void* w_v, void* image, int Lt, int Ht, int in_dim,
                                      int dt, int n_tile, cudaStream_t stream)
{
    const long long total = (long long)Lt * Ht * 2 * dt * in_dim / 8;
    const int threads = 256;
    tc_weight_relayout_kernel<<<(unsigned)((total + threads - 1) / threads), threads, 0, stream>>>(
        (const __nv_bfloat16*)w_k, (const __nv_bfloat16*)w_v, (uint8_t*)image, Lt, Ht, in_dim, dt, n_tile);
    return cudaGetLastError();
}

// programmatic stream serialization: see the kernel's griddepcontrol.wait
template <typename K>
static cudaError_t launch_pdl_span(K kernel, int grid, cudaStream_t stream, const TranslateParams& P, const TcLaunch& L)
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
    cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, P, L);
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_translate_tc(const TranslateParams& P, const TcConfig& cfg, int num_sms, cudaStream_t stream)
{
    TcLaunch L{};
    if (!tc_layout(P.in_dim, P.dt, P.ds, L)) return cudaErrorNotSupported;
    L.groups = P.Lt * P.Ht * 2 * L.n_split;
    L.seq_cached = P.batch <= kMaxSeqCache;
    L.m_tiles = (P.T_total + kTileM - 1) / kTileM;
    const long long UH = (long long)(L.groups / 2) * L.m_tiles;
    const int grid = (int)(UH < num_sms ? UH : num_sms);
    const int pp = L.in_dim / 64;
    switch (pp) {
    case 4:
        {
            static cudaError_t once = cudaFuncSetAttribute(translate_tc_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemMax);
            if (once != cudaSuccess) return once;
        }
        return launch_pdl_span(translate_tc_kernel<4>, grid, stream, P, L);
    case 2:
        {
            static cudaError_t once = cudaFuncSetAttribute(translate_tc_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemMax);
            if (once != cudaSuccess) return once;
        }
        return launch_pdl_span(translate_tc_kernel<2>, grid, stream, P, L);
    case 1:
        {
            static cudaError_t once = cudaFuncSetAttribute(translate_tc_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemMax);
            if (once != cudaSuccess) return once;
        }
        return launch_pdl_span(translate_tc_kernel<1>, grid, stream, P, L);
    default:
        return cudaErrorNotSupported;
    }
    (void)cfg;
    return cudaGetLastError();
}

}  // namespace kvx
