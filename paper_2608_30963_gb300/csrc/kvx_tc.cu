// kvx_tc.cu -- tensor-core translation kernel for sm_103a (tcgen05 / TMEM / bulk copies).
//
// The per-(target layer, target KV head, K|V) projection of T_theta (paper
// Section 5) is a dense [T x in] . [in x d_t] contraction; everything around it
// (span gather, RoPE undo, span mean, RoPE apply, cache write) is streaming work
// fused into the GEMM's prologue and epilogue.
//
// Persistent kernel, one CTA per SM.  Work unit = (target layer j, head set, K|V, output
// split(s), 128-token tile), where the head set holds the target heads that read the same
// input rows and fit one 512-column accumulator (the heads of a GQA expansion group, or every
// head in the dense per-layer form; one head otherwise): the unit's A (span means of the
// un-rotated source rows) is built once and multiplied by each (head, output split) "piece"
// of W into the piece's own accumulator slot.  A CTA walks an equal share of the K units and
// of the V units, group-major, so a one-piece unit's weight tile (B operand) stays in shared
// memory across its token tiles.  Warp roles:
//   warp 0      producer: resolves the spans of each 32-token sub-tile and, per
//               source head, copies the sub-tile's window of consecutive source
//               rows into a byte ring in shared memory with cp.async.bulk
//               (mbarrier transaction counts); loads a one-piece unit's whole B
//               image when it fits 64 KB, kept across the group's token tiles.
//   warp 1      lane 0, MMA: allocates TMEM, issues tcgen05.mma (M=128, N=n_tile,
//               K=16 steps over in, one source head's block of A at a time, one MMA
//               per piece) into a ring of fp32 accumulator slots.
//               lane 1, B-loader (streamed weights: several pieces per unit, or
//               inputs too wide to keep resident): one source head's rows of one
//               piece's W per (head-block, piece), through two slots.
//   warps 2-9   epilogue: tcgen05.ld the accumulator (one thread per token row,
//               two warps per TMEM lane quadrant), apply the target RoPE, round to
//               bf16, stage the row and write it to the target cache (contiguous
//               or paged) with cp.async.bulk, piece by piece.
//   warps 10-17 prologue: groups of d_s/16 lanes per target token, 16-byte
//               chunks per lane: undo the source RoPE of each span row, take the
//               span mean, round to bf16 and store A, one source head's block at
//               a time, in the UMMA K-major 128-byte-swizzled layout.
// Every wait is a bounded mbarrier poll: after ~1 s it records
// KVX_DEV_WAIT_TIMEOUT, raises a CTA-wide abort flag and the kernel drains and
// returns (no trap, no hang).
#include <climits>

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
constexpr int kBLoaderWarp = kXfWarp0 + kNumXfWarps;   // streams B pieces (streamed weights only)
constexpr int kThreads = (kBLoaderWarp + 1) * 32;
constexpr int kMaxSeqCache = 512;         // sequences whose metadata is kept in shared memory
constexpr int kMaxTcIn = 1024;            // widest translator input row (in) this kernel takes
constexpr int kMaxA = 2;                  // A head-block slots
constexpr int kMaxB = 2;                  // B slots (1: the group's whole image; 2: head-block pieces)
constexpr int kMaxD = 8;                  // accumulator slots in TMEM (512 columns / n_tile)
constexpr unsigned kBResidentMax = 65536; // largest B image kept resident per group
constexpr unsigned kBPieceMax = 32768;    // largest streamed B piece (one source head's rows)

// barrier indices
constexpr int kBarBFull = 0;               // +B slot
constexpr int kBarBEmpty = kBarBFull + kMaxB;
constexpr int kBarAFull = kBarBEmpty + kMaxB;   // +A slot
constexpr int kBarAEmpty = kBarAFull + kMaxA;
constexpr int kBarDFull = kBarAEmpty + kMaxA;   // +accumulator slot
constexpr int kBarDEmpty = kBarDFull + kMaxD;   // +accumulator slot
constexpr int kBarSlotFull = kBarDEmpty + kMaxD;    // +slot
constexpr int kBarSlotEmpty = kBarSlotFull + kNumSlots;
constexpr int kBarPair = kBarSlotEmpty + kNumSlots;   // +quad*2+{0,1}: the two epilogue warps of a quadrant meet
constexpr int kBarMmaDone = kBarPair + 8;             // after an abort: the issued MMAs have completed
constexpr int kNumBars = kBarMmaDone + 1;

// Span plan of one 32-token sub-tile, written by span_plan_kernel once per
// translation and read by every (layer, head, K|V) group of the tile:
//   header  {b0, c0, rows, 0}: the window of source rows [c0, c0 + rows) of sequence b0
//   entries {w0, lo, hi, b} x 32, longest span first: w0 = window row of the span
//           start (low 16 bits, signed; -1: read from global memory) | A row within
//           the sub-tile << 16 (0xFFFF: token past the end); [lo, hi) the clamped
//           source span of sequence b.

struct SpanEnt {
    int stage_row;   // window row of the span start; < 0: rows are read from global memory
    int lo, hi;      // source span within the sequence (hi <= lo: nothing to gather)
    int b;           // sequence
};

struct TcLaunch {
    int n_tile, n_split, in_dim, groups, m_tiles;
    int t_begin, t_end;          // target tokens of this launch
    const int4* plan_hdr;        // [sub-tiles of the launch]
    const int4* plan_ent;        // [sub-tiles][32]
    int r_heads;       // source heads per A row (in_dim / d_s)
    int n_a;           // A head-block slots (1 or 2)
    unsigned hb_bytes; // one A head-block: 128 rows x d_s bf16
    unsigned cap_rows; // most source rows one window may stage
    int n_slots;       // window slots of slot_bytes each
    int share;         // head units that read the same source rows, walked by interleaved CTA sets (1 = off)
    int hpu, spu;      // target heads and output splits of one work unit: all of them share the unit's
                       // A (its span-averaged input rows), each (head, split) is one piece with its own
                       // accumulator slot
    int np;            // pieces per unit: hpu * spu
    int nd;            // accumulator slots (ring over the pieces, in order)
    int n_b;           // B slots: 1 = the group's image stays resident across its tiles;
                       // 2 = streamed, one piece (one source head's rows of one piece's W) per
                       // (head-block, piece), by the B-loader lane
    unsigned b_bytes;  // one group's whole B image (in x n_tile bf16)
    unsigned b_slot_bytes;   // one B slot: b_bytes (resident) or ds x n_tile bf16 (streamed)
    unsigned row_bytes, stage_row_bytes, slot_bytes;
    unsigned off_b, off_a, off_stage, off_ring, off_meta, off_bar, off_misc, off_seq, off_turns;
    int seq_cached;   // per-sequence offsets and source lengths copied to shared memory
    unsigned idesc;
    unsigned tmem_cols;
};

struct Unit {
    int j, h, kv, nt, tile, g;   // first head and first split of the unit; g: B image of its first piece
};
// The CTA's units: an equal share of the K units, then of the V units (each share
// group-major, so a group's weights stay resident), walked with counters only.  A unit
// covers hpu consecutive target heads and spu consecutive output splits.
// When `share` > 1 head units read the same source rows (the heads of a GQA expansion group,
// or every head in the dense form, beyond those a unit covers), the CTAs form `share`
// interleaved sets: set i walks head unit i of every group, and CTA k of each set takes the
// k-th share of the same (layer, head group, tile) sequence.  The partners' reads of a window
// then come at about the same time, so the second one hits L2 instead of going back to DRAM.
struct Walker {
    int count, nK, it;
    int kv, j, h, nt, tile;
    int u0, v0, m_tiles, n_split, nsu, hpu, spu, Ht, E, hk, hv;
    Unit x;
    __device__ __forceinline__ void fill()
    {
        x.j = j; x.h = h; x.kv = kv; x.nt = nt * spu; x.tile = tile;
        x.g = ((j * Ht + h) * 2 + kv) * n_split + nt * spu;
    }
    __device__ __forceinline__ void seek(int idx, int kv_)
    {
        kv = kv_;
        const int hg = idx / m_tiles;
        tile = idx - hg * m_tiles;
        nt = hg % nsu;
        const int jq = hg / nsu;
        const int HtE = Ht / (hpu * E);
        h = (jq % HtE) * hpu * E + (kv ? hv : hk) * hpu;
        j = jq / HtE;
        fill();
    }
    __device__ __forceinline__ void start(const TcLaunch& L, int Ht_)
    {
        m_tiles = L.m_tiles; n_split = L.n_split; Ht = Ht_; E = L.share; hpu = L.hpu; spu = L.spu;
        nsu = n_split / spu;
        const long long UH = (long long)(L.groups / 2) * L.m_tiles / ((long long)E * hpu * spu);   // units of one set
        const int G = gridDim.x / E, c = blockIdx.x / E, vr = gridDim.x - 1 - (int)blockIdx.x;
        hk = (int)blockIdx.x % E;
        hv = vr % E;
        const int cv = vr / E;
        u0 = (int)((long long)c * UH / G);
        const int u1 = (int)((long long)(c + 1) * UH / G);
        v0 = (int)((long long)cv * UH / G);
        const int v1 = (int)((long long)(cv + 1) * UH / G);
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
            if (++nt == nsu) {
                nt = 0;
                if ((h += hpu * E) >= Ht) { h = (kv ? hv : hk) * hpu; ++j; }
            }
        }
        fill();
    }
    __device__ __forceinline__ bool last_of_group() const
    {
        return it + 1 == count || it + 1 == nK || tile + 1 == m_tiles;
    }
};

// B image of piece p of unit x: head x.h + p / spu, split x.nt + p % spu.
__device__ __forceinline__ int piece_group(const Unit& x, int p, int spu, int Ht, int n_split)
{
    const int hh = p / spu, s = p - hh * spu;
    return ((x.j * Ht + x.h + hh) * 2 + x.kv) * n_split + x.nt + s;
}

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

// Span bounds of target token tp as given (loaded ahead of use; identity: unused).
__device__ __forceinline__ int2 load_span(const TranslateParams& P, int tp)
{
    if (P.span_lo && tp < P.T_total) return make_int2(__ldg(&P.span_lo[tp]), __ldg(&P.span_hi[tp]));
    return make_int2(0, 0);
}

// Source-side resolution of one target token (sequence, clamped span) from its
// loaded span bounds.
__device__ __forceinline__ void resolve_src(const TranslateParams& P, const SeqView& sv, int tp, int2 span, int& b,
                                            int& lo, int& hi)
{
    b = sv.find(tp);
    const int t = tp - sv.off[b];
    int S = sv.slen[b];
    if (S > P.src_max_seq || S < 0) {
        set_status(P.status, KVX_DEV_SEQ_CLAMPED);
        S = S < 0 ? 0 : P.src_max_seq;
    }
    if (P.span_lo) { lo = span.x; hi = span.y; }
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
// DS: source head dim.  A is built one head-block (128 tokens x DS channels of one
// source head) at a time into a ring of n_a head-block slots, so the MMA of one
// head-block overlaps the build of the next.
// MULTI: units carry several pieces (shared A); false compiles the one-piece path with a ring of
// two accumulator slots and no piece loops.
template <int DS, bool MULTI>
__global__ void __launch_bounds__(kThreads, 1)
translate_tc_kernel(const __grid_constant__ TranslateParams P, const __grid_constant__ TcLaunch L)
{
    const int NP = MULTI ? L.np : 1;                       // pieces per unit
    const uint32_t ND = MULTI ? (uint32_t)L.nd : 2u;       // accumulator slots
    const int SPU = MULTI ? L.spu : 1;
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte aligned base, derived from smem_raw by pointer arithmetic so that the
    // compiler keeps every access below in the shared address space
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    uint8_t* sB = smem + L.off_b;
    uint8_t* sA = smem + L.off_a;
    uint8_t* sStage = smem + L.off_stage;
    uint8_t* sRing = smem + L.off_ring;
    int4* sMeta = reinterpret_cast<int4*>(smem + L.off_meta);
    uint64_t* sBar = reinterpret_cast<uint64_t*>(smem + L.off_bar);
    volatile int* sAbort = reinterpret_cast<volatile int*>(smem + L.off_misc);
    uint32_t* sTmemBase = reinterpret_cast<uint32_t*>(smem + L.off_misc + 4);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    auto bar = [&](int i) { return smem_u32(&sBar[i]); };

    if (threadIdx.x == 0) {
        *sAbort = 0;
        for (int i = 0; i < kMaxB; ++i) {
            mbar_init(bar(kBarBFull + i), 1);
            mbar_init(bar(kBarBEmpty + i), 1);
        }
        for (int i = 0; i < kMaxA; ++i) {
            mbar_init(bar(kBarAFull + i), kNumXfWarps);
            mbar_init(bar(kBarAEmpty + i), 1);
        }
        for (uint32_t i = 0; i < ND; ++i) {
            mbar_init(bar(kBarDFull + i), 1);
            mbar_init(bar(kBarDEmpty + i), kNumEpiWarps);
        }
        for (int i = 0; i < kNumSlots; ++i) {
            mbar_init(bar(kBarSlotFull + i), 1);
            mbar_init(bar(kBarSlotEmpty + i), kNumXfWarps);
        }
        for (int i = 0; i < 8; ++i) mbar_init(bar(kBarPair + i), 2);
        mbar_init(bar(kBarMmaDone), 1);
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

    const Waiter W{sAbort, P.status, P.wait_ns ? P.wait_ns : kWaitNs};
    const SeqView sv{L.seq_cached ? sSeqOff : P.seq_off, L.seq_cached ? sSrcLen : P.src_seq_len, P.batch};

    const int hw = L.n_tile >> 1;                 // pair half-width of an output split
    const int half_t = P.dt >> 1;

    if (warp == kProducerWarp) {
        // ------------------------------------------------------------ producer
        // Per 32-token sub-tile and source head: one window of consecutive source
        // rows [first span start, last span end) of the sub-tile's first sequence,
        // copied into the byte ring with one bulk copy.  Tokens whose span falls
        // outside the window (another sequence, a non-monotone span, a window cut at
        // the cap) are read by the prologue from global memory.
        // source rows read by more than one target head (repeated KV heads, dense form) stay in L2
        const uint64_t pol_src = (P.e > 1 || P.dense) ? policy_evict_last() : policy_evict_first();
        const uint64_t pol_keep = policy_evict_last();
        const bool rows_contig = P.ss == P.ds;
        const bool b_stream = L.n_b > 1;
        int cur_g = -1;
        uint32_t b_loads = 0, issued = 0;   // resident B images loaded (one slot); window copies issued
        // the group's whole B image into its slot (resident mode; streamed pieces come from the
        // B-loader lane)
        auto load_b = [&](const uint8_t* from, uint32_t bytes) -> bool {
            if (!W.wait(bar(kBarBEmpty), (b_loads & 1) ^ 1)) return false;
            if (lane == 0) mbar_arrive_expect_tx(bar(kBarBFull), bytes);
            __syncwarp();
            const uint32_t piece = bytes / 4;
            if (lane < 4)
                bulk_g2s(smem_u32(sB) + lane * piece, from + (size_t)lane * piece, piece, bar(kBarBFull), pol_keep);
            ++b_loads;
            return true;
        };
        int wslot = 0;             // window slot of the next window
        uint32_t wphase = 0;       // how often the slots have been cycled, mod 2
        bool ok = true;
        Walker wk;
        wk.start(L, P.Ht);
        // window headers of the current unit's sub-tiles (lane sq), loaded one unit ahead
        int4 hd = make_int4(0, 0, 0, 0);
        if (wk.more() && lane < kSubPerTile) hd = __ldg(L.plan_hdr + wk.x.tile * kSubPerTile + lane);
        for (; wk.more() && ok; wk.next()) {
            const Unit& x = wk.x;
            const uint8_t* img = (const uint8_t*)P.w + (size_t)x.g * L.b_bytes;
            if (!b_stream && x.g != cur_g) {
                if (!load_b(img, L.b_bytes)) { ok = false; break; }
                cur_g = x.g;
            }
            const int4 cur = hd;
            {
                Walker nx = wk;
                nx.next();
                if (nx.more() && lane < kSubPerTile) hd = __ldg(L.plan_hdr + nx.x.tile * kSubPerTile + lane);
            }
            for (int q = 0; q < L.r_heads && ok; ++q) {
                int src_slot, gq;
                head_block(P, x.j, x.h, q, src_slot, gq);
                const __nv_bfloat16* src = (const __nv_bfloat16*)(x.kv ? P.src_v[src_slot] : P.src_k[src_slot]);
#pragma unroll
                for (int sq = 0; sq < kSubPerTile; ++sq) {
                    if (!ok) break;
                    const int wb = __shfl_sync(0xffffffffu, cur.x, sq);
                    const int wlo = __shfl_sync(0xffffffffu, cur.y, sq);
                    const int wrows = __shfl_sync(0xffffffffu, cur.z, sq);
                    const int slot = wslot;
                    // the slot's previous window must have been released by the prologue warps
                    if (issued >= (uint32_t)L.n_slots && !W.wait(bar(kBarSlotEmpty + slot), wphase ^ 1)) {
                        ok = false;
                        break;
                    }
                    if (++wslot == L.n_slots) { wslot = 0; wphase ^= 1; }
                    const unsigned need = (unsigned)wrows * L.row_bytes;
                    const unsigned pos = (unsigned)slot * L.slot_bytes;
                    const uint32_t ring0 = smem_u32(sRing) + pos;
                    const __nv_bfloat16* s0 =
                        src + (long long)wb * P.sb + (long long)gq * P.sh + (long long)wlo * P.ss;
                    if (lane == 0) {
                        mbar_arrive_expect_tx(bar(kBarSlotFull + slot), need + (unsigned)(kSub * sizeof(int4)));
                        bulk_g2s(smem_u32(sMeta + slot * kSub), L.plan_ent + (size_t)(x.tile * kSubPerTile + sq) * kSub,
                                 (uint32_t)(kSub * sizeof(int4)), bar(kBarSlotFull + slot), pol_keep);
                        if (need && rows_contig) bulk_g2s(ring0, s0, need, bar(kBarSlotFull + slot), pol_src);
                    }
                    __syncwarp();
                    if (need && !rows_contig)
                        for (int r = lane; r < wrows; r += 32)
                            bulk_g2s(ring0 + (unsigned)r * L.row_bytes, s0 + (long long)r * P.ss, L.row_bytes,
                                     bar(kBarSlotFull + slot), pol_src);
                    ++issued;
                }
            }
        }
        // on abort, let copies already in flight land before the CTA leaves
        if (*sAbort) {
            const unsigned long long t0 = globaltimer();
            const uint32_t ns = (uint32_t)L.n_slots;
            for (uint32_t c = issued > ns ? issued - ns : 0; c < issued; ++c)
                while (!mbar_try_wait(bar(kBarSlotFull + c % ns), (c / ns) & 1) && globaltimer() - t0 < W.limit_ns) {}
            if (b_loads)
                while (!mbar_try_wait(bar(kBarBFull), (b_loads - 1) & 1) && globaltimer() - t0 < W.limit_ns) {}
        }
    } else if (warp == kMmaWarp) {
        const bool b_stream = L.n_b > 1;
        const uint32_t nb = (uint32_t)L.n_b, nd = ND;
        if (lane == 0) {
            // ------------------------------------------------------------ MMA issuer
            // Per unit and head-block q: one MMA per piece (head, output split) into the piece's
            // accumulator slot; the pieces' slots run as a ring of nd, in the order the epilogue
            // drains them.
            int cur_g = -1;
            uint32_t b_cnt = 0, pcount = 0, a_cnt = 0;   // B slot b_cnt % n_b, phase (b_cnt / n_b) & 1
            bool ok = true;
            Walker wk;
            for (wk.start(L, P.Ht); wk.more() && ok; wk.next()) {
                const Unit& x = wk.x;
                if (!b_stream && x.g != cur_g) {
                    if (!W.wait(bar(kBarBFull), b_cnt & 1)) break;
                    ++b_cnt;
                    cur_g = x.g;
                }
                for (int p = 0; p < NP && ok; ++p) {
                    const uint32_t c = pcount + (uint32_t)p;
                    if (!W.wait(bar(kBarDEmpty + c % nd), ((c / nd) & 1) ^ 1)) ok = false;
                }
                if (!ok) break;
                for (int q = 0; q < L.r_heads; ++q) {
                    const uint32_t sa = a_cnt % (uint32_t)L.n_a;
                    if (!W.wait(bar(kBarAFull + sa), (a_cnt / (uint32_t)L.n_a) & 1)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(sA) + sa * L.hb_bytes;
                    for (int p = 0; p < NP; ++p) {
                        // resident: the image's K-blocks of head-block q; streamed: the piece in its slot
                        uint32_t b0 = smem_u32(sB), kb0 = (uint32_t)q * (DS / 64);
                        const uint32_t bs = b_cnt % nb;
                        if (b_stream) {
                            if (!W.wait(bar(kBarBFull + bs), (b_cnt / nb) & 1)) { ok = false; break; }
                            tc_fence_after();
                            b0 += bs * L.b_slot_bytes;
                            kb0 = 0;
                        }
                        const uint32_t d = tmem_base + ((pcount + (uint32_t)p) % nd) * (uint32_t)L.n_tile;
#pragma unroll
                        for (int kk = 0; kk < DS / 16; ++kk) {
                            const uint32_t kb = kk >> 2, ko = (kk & 3) * 32;
                            const uint64_t ad = sw128_desc(a0 + kb * (kTileM * 128) + ko);
                            const uint64_t bd = sw128_desc(b0 + (kb0 + kb) * (L.n_tile * 128) + ko);
                            umma_bf16(d, ad, bd, L.idesc, (q > 0 || kk > 0) ? 1u : 0u);
                        }
                        if (b_stream) {
                            umma_commit(bar(kBarBEmpty + bs));
                            ++b_cnt;
                        }
                    }
                    if (!ok) break;
                    umma_commit(bar(kBarAEmpty + sa));
                    ++a_cnt;
                }
                if (!ok) break;
                for (int p = 0; p < NP; ++p) umma_commit(bar(kBarDFull + (pcount + (uint32_t)p) % nd));
                pcount += (uint32_t)NP;
                if (!b_stream && wk.last_of_group()) umma_commit(bar(kBarBEmpty));
            }
            if (*sAbort) {   // MMAs whose results nobody waited for must finish before TMEM is freed
                umma_commit(bar(kBarMmaDone));
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(bar(kBarMmaDone), 0) && globaltimer() - t0 < W.limit_ns) {}
            }
        }
        __syncwarp();
    } else if (warp == kBLoaderWarp) {
        const bool b_stream = L.n_b > 1;
        const uint32_t nb = (uint32_t)L.n_b;
        if (lane == 0 && b_stream) {
            // ------------------------------------------------------------ B-loader (streamed weights)
            // Per unit, head-block q and piece p, in the MMA's order: the d_s rows of head-block q of
            // the piece's B image (one source head's rows of W, n_tile output columns).
            const uint64_t pol_keep = policy_evict_last();
            uint32_t b_loads = 0;
            bool ok = true;
            Walker wk;
            for (wk.start(L, P.Ht); wk.more() && ok; wk.next()) {
                const Unit& x = wk.x;
                for (int q = 0; q < L.r_heads && ok; ++q)
                    for (int p = 0; p < NP; ++p) {
                        const uint32_t bs = b_loads % nb;
                        if (!W.wait(bar(kBarBEmpty + bs), ((b_loads / nb) & 1) ^ 1)) { ok = false; break; }
                        const uint8_t* img = (const uint8_t*)P.w +
                                             (size_t)piece_group(x, p, SPU, P.Ht, L.n_split) * L.b_bytes +
                                             (size_t)q * L.b_slot_bytes;
                        mbar_arrive_expect_tx(bar(kBarBFull + bs), L.b_slot_bytes);
                        bulk_g2s(smem_u32(sB) + bs * L.b_slot_bytes, img, L.b_slot_bytes, bar(kBarBFull + bs), pol_keep);
                        ++b_loads;
                    }
            }
            if (*sAbort) {   // let the copies in flight land before the CTA leaves
                const unsigned long long t0 = globaltimer();
                for (uint32_t c = b_loads > nb ? b_loads - nb : 0; c < b_loads; ++c)
                    while (!mbar_try_wait(bar(kBarBFull + c % nb), (c / nb) & 1) && globaltimer() - t0 < W.limit_ns) {}
            }
        }
        __syncwarp();
    } else if (warp >= kEpiWarp0 && warp < kEpiWarp0 + kNumEpiWarps) {
        // ------------------------------------------------------------ epilogue
        // Per unit: the output rows are resolved once; then per piece (head, output split), in
        // the MMA's order, the piece's accumulator slot is rotated, rounded, staged and stored.
        const int quad = warp & 3;
        const int half = (warp - kEpiWarp0) >> 2;          // which half of the rotary pairs
        const int m = quad * 32 + lane;
        const int pc_begin = half * (hw >> 1), pc_end = pc_begin + (hw >> 1);
        uint8_t* srow = sStage + (size_t)m * L.stage_row_bytes;
        const uint32_t srow_u32 = smem_u32(srow);
        const uint32_t nd = ND;
        uint32_t pcount = 0;
        bool ok = true;
        Walker wk;
        for (wk.start(L, P.Ht); wk.more() && ok; wk.next()) {
            const Unit& x = wk.x;
            // resolve the output row while the tile is still being computed
            const int tp = L.t_begin + x.tile * kTileM + m;
            const bool valid = tp < L.t_end;
            long long dst_off = -1;
            int pt = 0;
            if (valid) resolve_dst(P, sv, tp, dst_off, pt);
            const bool rot = x.kv == 0 && P.rt.enabled;
            for (int p = 0; p < NP; ++p, ++pcount) {
                const int hh = p / SPU, nt = x.nt + (p - hh * SPU);
                const uint32_t buf = pcount % nd;
                float2 cs[8];
                if (rot) rope_cs_vec<8>(sTurnT, pt, nt * hw + pc_begin, cs);
                if (!W.wait(bar(kBarDFull + buf), (pcount / nd) & 1)) { ok = false; break; }
                tc_fence_after();
                // the staging row is shared by the two warps of this quadrant; the row's
                // previous store must have read it
                bulk_wait_read0();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(kBarPair + quad * 2));
                if (!W.wait(bar(kBarPair + quad * 2), pcount & 1)) { ok = false; break; }
                const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + buf * (uint32_t)L.n_tile;
                for (int pc = pc_begin; pc < pc_end; pc += 8) {
                    float2 csn[8];
                    if (rot && pc + 8 < pc_end) rope_cs_vec<8>(sTurnT, pt, nt * hw + pc + 8, csn);
                    uint32_t r0[8], r1[8];
                    tmem_ld8(taddr + pc, r0);
                    tmem_ld8(taddr + hw + pc, r1);
                    tmem_ld_wait();
                    uint4 out0, out1;
                    // pair slots from rhalf on (partial rotary heads) do not rotate
                    rotate8_to_bf16(r0, r1, cs, rot && nt * hw + pc < P.rhalf_t, out0, out1);
                    if (rot) {
#pragma unroll
                        for (int e = 0; e < 8; ++e) cs[e] = csn[e];
                    }
                    *reinterpret_cast<uint4*>(srow + pc * 2) = out0;
                    *reinterpret_cast<uint4*>(srow + (hw + pc) * 2) = out1;
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(kBarDEmpty + buf));
                fence_proxy_async();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(kBarPair + quad * 2 + 1));
                if (!W.wait(bar(kBarPair + quad * 2 + 1), pcount & 1)) { ok = false; break; }
                // the quadrant's rows: stored by the half-0 warp when a unit has one piece, split
                // between the two warps by lane parity when it has several
                if ((NP > 1 ? (lane & 1) == half : half == 0) && valid && dst_off >= 0) {
                    __nv_bfloat16* dst = (__nv_bfloat16*)(x.kv ? P.dst_v[x.j] : P.dst_k[x.j]) + dst_off +
                                         dst_head_off(P, x.h + hh);
                    if (P.plain_stores) {
                        store_row_slots_plain(dst, srow, nt * hw, hw, half_t, P.rhalf_t);
                    } else {
                        store_row_slots(dst, srow_u32, nt * hw, hw, half_t, P.rhalf_t);
                        bulk_commit();
                    }
                }
            }
        }
        bulk_wait0();
    } else if (warp >= kXfWarp0 && warp < kXfWarp0 + kNumXfWarps) {
        // ------------------------------------------------------------ prologue (A head-blocks)
        // Lanes split into groups of LPT, one target token per group; a lane owns one
        // chunk pair: pair slots [8cp, 8cp+8), i.e. channels [8cp, 8cp+8) and their rotary
        // partners [DS/2+8cp, ...) (pair_channels: a partial rotary head pairs at rhalf,
        // and lanes past rhalf hold channels that do not rotate), so each source row is read
        // as two 16-byte loads per lane (a group reads whole 128-byte row segments: no bank
        // conflicts on the linear window rows) and A is written at the same channels.
        constexpr int LPT = DS / 16;
        constexpr int TPW = 32 / LPT;
        constexpr int HALF = DS / 2;
        const int tw = warp - kXfWarp0;
        const int cp = lane % LPT;
        const int u = lane / LPT;
        int k_lo, k_hi;
        pair_channels(8 * cp, HALF, P.rhalf_s, k_lo, k_hi);
        const bool lane_rot = 8 * cp < P.rhalf_s;
        const uint32_t c_lo = (uint32_t)k_lo * 2, c_hi = (uint32_t)k_hi * 2;
        const uint32_t a_lo = (uint32_t)(k_lo >> 6) * (kTileM * 128), a_hi = (uint32_t)(k_hi >> 6) * (kTileM * 128);
        const int ch_lo = (k_lo >> 3) & 7, ch_hi = (k_hi >> 3) & 7;
        unsigned long long turn[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) turn[e] = sTurnS[cp * 8 + e];
        uint32_t a_cnt = 0;
        int wslot = 0;
        uint32_t wphase = 0;
        bool ok = true;
        Walker wk;
        for (wk.start(L, P.Ht); wk.more() && ok; wk.next()) {
            const Unit& x = wk.x;
            const bool rot = x.kv == 0 && P.rs.enabled && lane_rot;
            for (int q = 0; q < L.r_heads && ok; ++q) {
                int src_slot, gq;
                head_block(P, x.j, x.h, q, src_slot, gq);
                const __nv_bfloat16* src = (const __nv_bfloat16*)(x.kv ? P.src_v[src_slot] : P.src_k[src_slot]);
                const uint32_t sa = a_cnt % (uint32_t)L.n_a;
                if (!W.wait(bar(kBarAEmpty + sa), ((a_cnt / (uint32_t)L.n_a) & 1) ^ 1)) { ok = false; break; }
                uint8_t* sAq = sA + sa * L.hb_bytes;
                for (int sq = 0; sq < kSubPerTile; ++sq) {
                    const int slot = wslot;
                    if (!W.wait(bar(kBarSlotFull + slot), wphase)) { ok = false; break; }
                    if (++wslot == L.n_slots) { wslot = 0; wphase ^= 1; }
                    const uint8_t* ring = sRing + (size_t)slot * L.slot_bytes;
                    // entries are sorted by span length; the warp's chunk of them rotates with
                    // the sub-tile so that long spans spread over the warps
                    for (int tt = ((tw + 2 * sq) & (kNumXfWarps - 1)) * TPW + u; tt < kSub; tt += kNumXfWarps * TPW) {
                        const int4 ent = sMeta[slot * kSub + tt];
                        const int row_in = (int)((unsigned)ent.x >> 16);
                        if (row_in >= kSub) continue;   // token past the end
                        const int row = sq * kSub + row_in;
                        const SpanEnt m{(int)(short)(ent.x & 0xFFFF), ent.y, ent.z, ent.w};
                        const int n = max(m.hi - m.lo, 0);
                        float a0[8], a1[8];
#pragma unroll
                        for (int e = 0; e < 8; ++e) { a0[e] = 0.f; a1[e] = 0.f; }
                        for (int o = 0; o < n; ++o) {
                            uint4 w0, w1;
                            if (m.stage_row >= 0) {
                                const uint8_t* rp = ring + (size_t)(m.stage_row + o) * (DS * 2);
                                w0 = *reinterpret_cast<const uint4*>(rp + c_lo);
                                w1 = *reinterpret_cast<const uint4*>(rp + c_hi);
                            } else {
                                const uint8_t* rp = reinterpret_cast<const uint8_t*>(
                                    src + (long long)m.b * P.sb + (long long)gq * P.sh +
                                    (long long)(m.lo + o) * P.ss);
                                w0 = __ldg(reinterpret_cast<const uint4*>(rp + c_lo));
                                w1 = __ldg(reinterpret_cast<const uint4*>(rp + c_hi));
                            }
                            const uint32_t v0[4] = {w0.x, w0.y, w0.z, w0.w}, v1[4] = {w1.x, w1.y, w1.z, w1.w};
                            if (rot) {
                                const int pos = src_pos_of(P, m.b, m.lo + o);
#pragma unroll
                                for (int k = 0; k < 4; ++k) {   // undo the rotation: R(-theta)
                                    const float2 ca = turn_cs(turn[2 * k], pos), cb = turn_cs(turn[2 * k + 1], pos);
                                    if (o == 0) {
                                        unrotate1(bf_lo(v0[k]), bf_lo(v1[k]), ca, a0[2 * k], a1[2 * k]);
                                        unrotate1(bf_hi(v0[k]), bf_hi(v1[k]), cb, a0[2 * k + 1], a1[2 * k + 1]);
                                    } else {
                                        unrotate_acc(bf_lo(v0[k]), bf_lo(v1[k]), ca, a0[2 * k], a1[2 * k]);
                                        unrotate_acc(bf_hi(v0[k]), bf_hi(v1[k]), cb, a0[2 * k + 1], a1[2 * k + 1]);
                                    }
                                }
                            } else {
#pragma unroll
                                for (int k = 0; k < 4; ++k) {
                                    a0[2 * k] += bf_lo(v0[k]);
                                    a0[2 * k + 1] += bf_hi(v0[k]);
                                    a1[2 * k] += bf_lo(v1[k]);
                                    a1[2 * k + 1] += bf_hi(v1[k]);
                                }
                            }
                        }
                        // span mean; 1/n is exact for n = 1, 2 (the common spans)
                        const float inv_n = n > 0 ? __frcp_rn((float)n) : 0.f;
                        uint32_t o0[4], o1[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            o0[k] = pack_bf16(a0[2 * k] * inv_n, a0[2 * k + 1] * inv_n);
                            o1[k] = pack_bf16(a1[2 * k] * inv_n, a1[2 * k + 1] * inv_n);
                        }
                        const uint32_t r7 = (uint32_t)(row & 7);
                        *reinterpret_cast<uint4*>(sAq + a_lo + row * 128 + (((uint32_t)ch_lo ^ r7) << 4)) =
                            make_uint4(o0[0], o0[1], o0[2], o0[3]);
                        *reinterpret_cast<uint4*>(sAq + a_hi + row * 128 + (((uint32_t)ch_hi ^ r7) << 4)) =
                            make_uint4(o1[0], o1[1], o1[2], o1[3]);
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(bar(kBarSlotEmpty + slot));
                }
                if (!ok) break;
                fence_proxy_async();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar(kBarAFull + sa));
                ++a_cnt;
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, L.tmem_cols);
    }
}

// Span plan of the sub-tiles of target tokens [t_begin, t_end): one warp per
// 32-token sub-tile, one lane per token (layout: see the comment at the top).  Every
// sub-tile of the launch's 128-token tiles gets a header and 32 entries; those past
// the end get an empty window and entries marked past the end.
__global__ void __launch_bounds__(128) span_plan_kernel(const __grid_constant__ TranslateParams P, int t_begin,
                                                        int t_end, int cap_rows, int4* __restrict__ hdr,
                                                        int4* __restrict__ ent)
{
    // the previous launch in the stream may still read the plan buffer
    grid_dependency_wait();
    grid_launch_dependents();
    const int sub = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    const int nsub = (t_end - t_begin + kTileM - 1) / kTileM * kSubPerTile;
    if (sub >= nsub) return;
    const SeqView sv{P.seq_off, P.src_seq_len, P.batch};
    const int tp = t_begin + sub * kSub + lane;
    const bool valid = tp < t_end;
    int b = -1, lo = 0, hi = 0;
    if (valid) resolve_src(P, sv, tp, load_span(P, tp), b, lo, hi);
    // valid tokens are a prefix of the sub-tile, so lane 0 opens the window
    const int b0 = __shfl_sync(0xffffffffu, b, 0);
    const int c0 = __shfl_sync(0xffffffffu, lo, 0);
    const bool same = valid && b == b0;
    const int hmax = __reduce_max_sync(0xffffffffu, same ? hi : INT_MIN);
    int R = hmax == INT_MIN ? 0 : max(hmax - c0, 0);
    R = min(R, cap_rows);
    const bool inwin = same && lo >= c0 && hi <= c0 + R;
    const int stage_row = inwin ? lo - c0 : -1;
    // rank: longest span first (lengths above 3 share a bucket), then lane order;
    // tokens past the end last
    const int key = valid ? min(max(hi - lo, 0), 3) : -1;
    int rank = 0;
#pragma unroll
    for (int k = 3; k >= -1; --k) {
        const unsigned bal = __ballot_sync(0xffffffffu, key == k);
        if (k > key) rank += __popc(bal);
        else if (k == key) rank += __popc(bal & ((1u << lane) - 1u));
    }
    const int w0 = (int)(((unsigned)stage_row & 0xFFFFu) | ((valid ? (unsigned)lane : 0xFFFFu) << 16));
    ent[(size_t)sub * kSub + rank] = make_int4(w0, lo, hi, b < 0 ? 0 : b);
    if (lane == 0) hdr[sub] = make_int4(b0 < 0 ? 0 : b0, c0, R, 0);
}

// Weight images: for group g = ((j*Ht + h)*2 + kv)*n_split + nt, the B operand
// [n_tile rows = output columns][in] in K-major SW128 layout.  Image row n holds pair
// slot k = nt*hw + (n mod hw): its first channel for n < hw, its partner above
// (pair_channels: (k, k + d_t/2), or the partial rotary pairing), so an image holds
// whole RoPE pairs and the epilogue rotates columns n and n + hw together.
__global__ void tc_weight_relayout_kernel(const __nv_bfloat16* __restrict__ wk, const __nv_bfloat16* __restrict__ wv,
                                          uint8_t* __restrict__ img, int Lt, int Ht, int in_dim, int dt, int n_tile,
                                          int rhalf_t)
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
    int c_lo, c_hi;
    pair_channels(nt * hw + (n < hw ? n : n - hw), dt / 2, rhalf_t, c_lo, c_hi);
    const int col = n < hw ? c_lo : c_hi;
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

// share: target heads that read the same input rows (the heads of a GQA expansion group, or
// every head in the dense form; 1 otherwise).
bool tc_layout(int in_dim, int dt, int ds, int share, TcLaunch& L)
{
    if (in_dim % 64 || in_dim > kMaxTcIn || in_dim < 64) return false;
    if (dt != 64 && dt != 128 && dt != 256) return false;
    if (ds != 64 && ds != 128 && ds != 256) return false;
    if (in_dim % ds) return false;
    L.in_dim = in_dim;
    L.r_heads = in_dim / ds;
    // Heads per unit: as many of the heads sharing the input rows as the 512 accumulator columns
    // hold (d_t each), so their A is built once; each (head, output split) is a piece, and the
    // pieces' weights stream through two slots, one head-block (ds x n_tile) at a time.
    // Only when one piece covers a whole output head (ds x dt weights within a streamed slot):
    // splitting the heads' rows into narrower pieces multiplies the row stores.
    int hpu = 1;
    if ((unsigned)(ds * dt * 2) <= kBPieceMax)
        for (int c = share; c > 1; --c)
            if (share % c == 0 && c * dt <= 512) { hpu = c; break; }
    if (hpu > 1) {
        L.n_b = kMaxB;
        L.n_tile = dt;
        while ((unsigned)(ds * L.n_tile * 2) > kBPieceMax && L.n_tile > 64) L.n_tile >>= 1;
        L.n_split = dt / L.n_tile;
        L.hpu = hpu;
        L.spu = L.n_split;
        L.nd = 512 / L.n_tile;
    } else {
        // one head per unit: B resident per group while one output split's image fits
        // kBResidentMax; beyond that, streamed one head-block piece (ds x n_tile) at a time
        L.n_tile = dt;
        while ((unsigned)(in_dim * L.n_tile * 2) > kBResidentMax && L.n_tile > 64 && in_dim <= 256) L.n_tile >>= 1;
        L.n_b = (unsigned)(in_dim * L.n_tile * 2) <= kBResidentMax ? 1 : kMaxB;
        if (L.n_b > 1) {
            L.n_tile = dt;
            while ((unsigned)(ds * L.n_tile * 2) > kBPieceMax && L.n_tile > 64) L.n_tile >>= 1;
        }
        L.n_split = dt / L.n_tile;
        L.hpu = 1;
        L.spu = 1;
        L.nd = 2;
    }
    L.np = L.hpu * L.spu;
    if (L.nd > kMaxD || L.np > L.nd) return false;
    L.b_bytes = (unsigned)(in_dim * L.n_tile * 2);
    L.b_slot_bytes = L.n_b > 1 ? (unsigned)(ds * L.n_tile * 2) : L.b_bytes;
    L.hb_bytes = (unsigned)(kTileM * ds * 2);
    L.row_bytes = (unsigned)(ds * 2);
    L.stage_row_bytes = (unsigned)(L.n_tile * 2 + 16);
    // Window slots of 48 source rows: a 32-token sub-tile of spans averaging 1.3
    // tokens needs ~42; tokens whose rows fall past the cap are read from global
    // memory.  Two A slots when four window slots still fit, else one.
    L.cap_rows = 48;
    L.slot_bytes = L.cap_rows * L.row_bytes;
    for (int n_a = kMaxA; n_a >= 1; --n_a) {
        unsigned off = 0;
        auto take = [&](unsigned bytes, unsigned align) {
            off = (off + align - 1) / align * align;
            const unsigned o = off;
            off += bytes;
            return o;
        };
        L.n_a = n_a;
        L.off_b = take((unsigned)L.n_b * L.b_slot_bytes, 1024);
        L.off_a = take((unsigned)n_a * L.hb_bytes, 1024);
        L.off_stage = take(kTileM * L.stage_row_bytes, 128);
        L.off_meta = take(kNumSlots * kSub * sizeof(int4), 16);
        L.off_bar = take(kNumBars * 8, 8);
        L.off_misc = take(16, 16);
        L.off_seq = take((2 * kMaxSeqCache + 1) * sizeof(int), 16);
        L.off_turns = take((unsigned)(ds / 2 + dt / 2) * 8, 16);
        L.off_ring = (off + 127) / 128 * 128;
        const int avail = kSmemMax - 1024 - (int)L.off_ring;   // 1024: alignment slack of the dynamic base
        const int slots = avail > 0 ? (int)((unsigned)avail / L.slot_bytes) : 0;
        L.n_slots = slots < kNumSlots ? slots : kNumSlots;
        if (L.n_slots >= (n_a > 1 ? 4 : 2)) break;
        if (n_a == 1) return false;
    }
    L.idesc = make_idesc(kTileM, L.n_tile);
    unsigned cols = 32;
    while (cols < (unsigned)L.nd * (unsigned)L.n_tile) cols <<= 1;
    L.tmem_cols = cols;
    return cols <= 512;
}

}  // namespace

TcConfig tc_config(int in_dim, int dt, int ds, int share)
{
    TcLaunch L{};
    TcConfig c{0, 0, 0, kThreads, 0};
    if (!tc_layout(in_dim, dt, ds, share, L)) return c;
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
                                      int dt, int n_tile, int rhalf_t, cudaStream_t stream)
{
    const long long total = (long long)Lt * Ht * 2 * dt * in_dim / 8;
    const int threads = 256;
    tc_weight_relayout_kernel<<<(unsigned)((total + threads - 1) / threads), threads, 0, stream>>>(
        (const __nv_bfloat16*)w_k, (const __nv_bfloat16*)w_v, (uint8_t*)image, Lt, Ht, in_dim, dt, n_tile, rhalf_t);
    return cudaGetLastError();
}

// programmatic stream serialization: see the kernels' griddepcontrol.wait
template <typename K, typename... Args>
static cudaError_t launch_pdl(K kernel, int grid, int threads, size_t smem, cudaStream_t stream, Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, args...);
    return e != cudaSuccess ? e : cudaGetLastError();
}

template <int DS, bool MULTI>
static cudaError_t launch_span_ds(int grid, cudaStream_t stream, const TranslateParams& P, const TcLaunch& L)
{
    const cudaError_t e = smem_opt_in<translate_tc_kernel<DS, MULTI>>(kSmemMax);
    if (e != cudaSuccess) return e;
    // the B-loader warp (the last one) only when the weights stream
    const int threads = L.n_b > 1 ? kThreads : kThreads - 32;
    return launch_pdl(translate_tc_kernel<DS, MULTI>, grid, threads, kSmemMax, stream, P, L);
}
template <int DS>
static cudaError_t launch_span(int grid, cudaStream_t stream, const TranslateParams& P, const TcLaunch& L)
{
    return L.np > 1 ? launch_span_ds<DS, true>(grid, stream, P, L) : launch_span_ds<DS, false>(grid, stream, P, L);
}

size_t tc_plan_bytes(int tokens)
{
    const size_t nsub = (size_t)(tokens + kSub - 1) / kSub;
    return nsub * sizeof(int4) * (1 + kSub);
}

void tc_plan_layout(int T_total, int plan_tokens, int* nsub, int* ent_off)
{
    const int chunk = plan_tokens / kTileM * kTileM;
    *ent_off = (chunk + kSub - 1) / kSub;
    *nsub = 0;
    if (chunk <= 0 || T_total <= 0) return;
    const int last = (T_total - 1) / chunk * chunk;   // first token of the last chunk
    *nsub = (T_total - last + kTileM - 1) / kTileM * kSubPerTile;
}

cudaError_t launch_translate_tc(const TranslateParams& P, const TcConfig& cfg, int num_sms, void* plan,
                                int plan_tokens, cudaStream_t stream, int* launches)
{
    *launches = 0;
    TcLaunch L{};
    if (!tc_layout(P.in_dim, P.dt, P.ds, share_heads(P), L)) return cudaErrorNotSupported;
    if (P.ds != 64 && P.ds != 128 && P.ds != 256) return cudaErrorNotSupported;
    L.groups = P.Lt * P.Ht * 2 * L.n_split;
    L.seq_cached = P.batch <= kMaxSeqCache;
    const int chunk = plan_tokens / kTileM * kTileM;
    if (chunk <= 0 || !plan) return cudaErrorInvalidValue;
    int4* hdr = reinterpret_cast<int4*>(plan);
    int4* ent = hdr + (chunk + kSub - 1) / kSub;
    // one plan + one translation launch per chunk of at most plan_tokens target tokens
    for (int t0 = 0; t0 < P.T_total; t0 += chunk) {
        const int t1 = P.T_total - t0 < chunk ? P.T_total : t0 + chunk;
        L.t_begin = t0;
        L.t_end = t1;
        L.m_tiles = (t1 - t0 + kTileM - 1) / kTileM;
        L.plan_hdr = hdr;
        L.plan_ent = ent;
        const int nsub = L.m_tiles * kSubPerTile;
        cudaError_t e = launch_pdl(span_plan_kernel, (nsub + 3) / 4, 128, 0, stream, P, t0, t1, (int)L.cap_rows, hdr, ent);
        if (e != cudaSuccess) return e;
        ++*launches;
        const long long UH = (long long)(L.groups / 2) * L.m_tiles / (L.hpu * L.spu);
        const int grid = (int)(UH < num_sms ? UH : num_sms);
        // head units that share source rows beyond the heads one unit covers (a GQA expansion
        // group, or all heads of the dense form): interleaved CTA sets
        const int E = share_heads(P) / L.hpu;
        L.share = E > 1 && P.Ht % (E * L.hpu) == 0 && grid % E == 0 ? E : 1;
        switch (P.ds) {
        case 256: e = launch_span<256>(grid, stream, P, L); break;
        case 128: e = launch_span<128>(grid, stream, P, L); break;
        default: e = launch_span<64>(grid, stream, P, L); break;
        }
        if (e != cudaSuccess) return e;
        ++*launches;
    }
    (void)cfg;
    return cudaSuccess;
}

}  // namespace kvx
