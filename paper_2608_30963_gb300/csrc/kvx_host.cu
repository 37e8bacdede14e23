// kvx_host.cu -- host side of the kvx C ABI: validation, translator state,
// weight upload and re-layout, RoPE tables, launch selection, error status.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <mutex>
#include <string>
#include <vector>

#include "kvx_common.cuh"
#include "kvx_kernels.h"

using namespace kvx;

struct kvx_translator {
    Geometry geo;                       // validated description (shared with the fitter)
    kvx_translator_desc desc;
    int layer_map[KVX_MAX_SRC_SLOTS];   // [j * kl + k]: source layers of target layer j
    int device = 0;
    int num_sms = 0;
    int in_dim = 0, r = 1, e = 1;
    int dense = 0, kl = 1, hpl = 1;     // form, source layers per target layer, heads per layer block
    int path = KVX_PATH_SIMT;
    int max_position = 0;
    void* w = nullptr;           // SIMT: [2][Lt][Ht][in][out] dtype; tcgen05: pre-swizzled images
    size_t w_bytes = 0;
    unsigned long long* rope = nullptr;   // fixed-point turns: source [d_s/2] | target [d_t/2]
    unsigned long long host_turns[256];   // host copy of the same
    size_t rope_bytes = 0;
    RopeTable rs{}, rt{};
    int rope_same = 0;           // source and target turns identical (same d, same frequencies)
    unsigned* status = nullptr;
    TcConfig tc{};
    // span plan of the tensor-core span kernel: sub-tile windows and per-token entries
    // for up to kPlanTokens target tokens per launch (longer calls run in chunks)
    static constexpr int kPlanTokens = 1 << 16;
    void* plan = nullptr;
    int last_launches = 0;       // kernel launches of the most recent kvx_translate
    int last_span_tokens = 0;    // target tokens of the most recent call if it ran the span kernel, else 0
    int dbg_stall_unit1 = 0;     // kvx_debug_stall_next_translate, for the next call only
    unsigned long long dbg_wait_ns = 0;
    // encoded source tensor maps of the identity-alignment kernel, a few per (target layer, K|V)
    struct MapEntry {
        const void* ptr = nullptr;
        int S = 0, B = 0;
        long long ss = 0, sh = 0, sb = 0;
        unsigned long long stamp = 0;
        alignas(64) unsigned char map[128];
    };
    static constexpr int kMapWays = 4;
    std::vector<MapEntry> maps;
    unsigned long long map_stamp = 0;
};

// Encoded tensor map for the source K or V cache of target layer j (cached by
// pointer, length, batch and strides).  Returns nullptr if encoding fails.
static const void* source_map(kvx_translator* t, int j, int kv, const void* ptr, const kvx_src_kv* src)
{
    const int slot = (j * 2 + kv) * kvx_translator::kMapWays;
    kvx_translator::MapEntry* lru = nullptr;
    for (int w = 0; w < kvx_translator::kMapWays; ++w) {
        kvx_translator::MapEntry& e = t->maps[slot + w];
        if (e.ptr == ptr && e.S == src->max_seq && e.B == src->batch && e.ss == src->stride_s &&
            e.sh == src->stride_h && e.sb == src->stride_b) {
            e.stamp = ++t->map_stamp;
            return e.map;
        }
        if (!lru || e.stamp < lru->stamp) lru = &e;
    }
    if (!encode_source_map(lru->map, ptr, t->desc.src.head_dim, src->max_seq, t->desc.src.num_kv_heads, src->batch,
                           src->stride_s, src->stride_h, src->stride_b))
        return nullptr;
    lru->ptr = ptr;
    lru->S = src->max_seq;
    lru->B = src->batch;
    lru->ss = src->stride_s;
    lru->sh = src->stride_h;
    lru->sb = src->stride_b;
    lru->stamp = ++t->map_stamp;
    return lru->map;
}

static thread_local std::string g_last_error;

static kvx_status fail(kvx_status s, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
static kvx_status fail(kvx_status s, const char* fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return s;
}

#define CUDA_OR_FAIL(call)                                                                       \
    do {                                                                                         \
        cudaError_t e_ = (call);                                                                 \
        if (e_ != cudaSuccess)                                                                   \
            return fail(KVX_ERR_CUDA, "%s: %s (%s:%d)", #call, cudaGetErrorString(e_), __FILE__, \
                        __LINE__);                                                               \
    } while (0)

static bool head_dim_ok(int d) { return d == 64 || d == 128 || d == 256; }

extern "C" KVX_API const char* kvx_last_error(void) { return g_last_error.c_str(); }

extern "C" KVX_API kvx_status kvx_layer_map_nearest(int32_t Ls, int32_t Lt, int32_t* out)
{
    if (Ls < 1 || Lt < 1 || !out) return fail(KVX_ERR_INVALID_ARG, "layer_map_nearest: bad arguments");
    for (int j = 0; j < Lt; ++j) {
        if (Lt == 1) { out[j] = 0; continue; }
        // round(j (Ls-1) / (Lt-1)), halves up, in exact integers
        const long long num = 2LL * j * (Ls - 1) + (Lt - 1);
        out[j] = (int32_t)(num / (2LL * (Lt - 1)));
    }
    return KVX_OK;
}

static void free_translator(kvx_translator* t)
{
    if (!t) return;
    if (t->w) cudaFree(t->w);
    if (t->rope) cudaFree(t->rope);
    if (t->status) cudaFree(t->status);
    if (t->plan) cudaFree(t->plan);
    delete t;
}

namespace kvx {

void set_last_error(const char* msg) { g_last_error = msg; }

kvx_status make_geometry(const kvx_translator_desc* desc, const char* who, Geometry& g, char* err)
{
    auto bad = [&](kvx_status st, const char* fmt, auto... args) {
        int n = snprintf(err, 512, "%s: ", who);
        snprintf(err + n, 512 - n, fmt, args...);
        return st;
    };
    const kvx_model_geom& s = desc->src;
    const kvx_model_geom& d = desc->dst;
    if (s.num_layers < 1 || d.num_layers < 1 || s.num_kv_heads < 1 || d.num_kv_heads < 1)
        return bad(KVX_ERR_INVALID_ARG, "layer and head counts must be >= 1");
    if (d.num_layers > KVX_MAX_TARGET_LAYERS)
        return bad(KVX_ERR_UNSUPPORTED, "at most %d target layers", KVX_MAX_TARGET_LAYERS);
    if (!head_dim_ok(s.head_dim) || !head_dim_ok(d.head_dim))
        return bad(KVX_ERR_UNSUPPORTED, "head dims must be 64, 128 or 256 (got %d, %d)", s.head_dim, d.head_dim);
    if (s.num_kv_heads % d.num_kv_heads != 0 && d.num_kv_heads % s.num_kv_heads != 0)
        return bad(KVX_ERR_UNSUPPORTED, "neither KV head count divides the other (%d, %d)", s.num_kv_heads,
                   d.num_kv_heads);
    if (desc->dtype != KVX_BF16 && desc->dtype != KVX_FP32)
        return bad(KVX_ERR_INVALID_ARG, "unknown dtype %d", desc->dtype);
    if (desc->path < KVX_PATH_AUTO || desc->path > KVX_PATH_TCGEN05)
        return bad(KVX_ERR_INVALID_ARG, "unknown path %d", desc->path);
    if (!rope_schedule_ok(s) || !rope_schedule_ok(d))
        return bad(KVX_ERR_INVALID_ARG, "unknown rope_type, schedule parameters out of range or rotary_dim "
                                        "not 0 or a multiple of 16 in [16, head_dim] (source type %d rotary_dim "
                                        "%d, target type %d rotary_dim %d)", s.rope_type, s.rotary_dim, d.rope_type,
                   d.rotary_dim);
    const int max_pos = desc->max_position ? desc->max_position : (1 << 24);
    if (max_pos < 1 || max_pos > (1 << 30)) return bad(KVX_ERR_INVALID_ARG, "max_position must be in [1, 1<<30]");
    if (desc->form != KVX_FORM_GROUPED && desc->form != KVX_FORM_DENSE)
        return bad(KVX_ERR_INVALID_ARG, "unknown form %d", desc->form);
    const int kl = desc->layers_per_target > 1 ? desc->layers_per_target : 1;
    if (desc->layers_per_target < 0 || kl > 4 || d.num_layers * kl > KVX_MAX_SRC_SLOTS)
        return bad(KVX_ERR_INVALID_ARG, "layers_per_target %d outside [0, 4] or more than %d "
                                        "(target layer, source layer) pairs", desc->layers_per_target, KVX_MAX_SRC_SLOTS);
    if (kl > 1 && !desc->layer_map) return bad(KVX_ERR_INVALID_ARG, "layers_per_target > 1 needs an explicit layer_map");
    g.desc = *desc;
    g.desc.layer_map = nullptr;
    g.max_position = max_pos;
    g.kl = kl;
    g.dense = desc->form == KVX_FORM_DENSE;
    if (desc->layer_map) {
        for (int i = 0; i < d.num_layers * kl; ++i) {
            if (desc->layer_map[i] < 0 || desc->layer_map[i] >= s.num_layers)
                return bad(KVX_ERR_INVALID_ARG, "layer_map[%d] = %d outside [0, %d)", i, desc->layer_map[i],
                           s.num_layers);
            g.layer_map[i] = desc->layer_map[i];
        }
    } else {
        kvx_layer_map_nearest(s.num_layers, d.num_layers, g.layer_map);
    }
    g.r = g.e = 1;
    if (s.num_kv_heads >= d.num_kv_heads) g.r = s.num_kv_heads / d.num_kv_heads;
    else g.e = d.num_kv_heads / s.num_kv_heads;
    g.hpl = g.dense ? s.num_kv_heads : g.r;
    g.in_dim = kl * g.hpl * s.head_dim;
    if (g.in_dim > 1024) return bad(KVX_ERR_UNSUPPORTED, "translator input width %d > 1024", g.in_dim);
    // rotation frequencies as fixed-point turns (kvx_common.cuh)
    const int hs = s.head_dim / 2, hd = d.head_dim / 2;
    auto fill = [&](const kvx_model_geom& m, unsigned long long* o) {   // pairs past rotary_dim/2: 0
        for (int i = 0; i < rope_rot_dim(m) / 2; ++i)
            o[i] = m.rope_base <= 0.0 ? 0ull : (unsigned long long)ldexp(rope_inv_freq(m, i) / (2.0 * M_PI), 64);
    };
    memset(g.turns, 0, sizeof g.turns);
    fill(s, g.turns);
    fill(d, g.turns + hs);
    // the two rotations coincide when head dims, rotating channels, enablement and every frequency agree
    g.rope_same = hs == hd && rope_rot_dim(s) == rope_rot_dim(d) && (s.rope_base > 0.0) == (d.rope_base > 0.0) &&
                  memcmp(g.turns, g.turns + hs, (size_t)hs * sizeof(unsigned long long)) == 0;
    return KVX_OK;
}

static bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

kvx_status make_params(const Geometry& g, const unsigned long long* dev_turns, unsigned* status, const void* w,
                       const kvx_src_kv* src, const kvx_tgt_tokens* tgt, const kvx_dst_kv* dst, TranslateParams& P,
                       const char* who, char* err)
{
    auto bad = [&](kvx_status st, const char* fmt, auto... args) {
        int n = snprintf(err, 512, "%s: ", who);
        snprintf(err + n, 512 - n, fmt, args...);
        return st;
    };
    const kvx_translator_desc& D = g.desc;
    const int Lt = D.dst.num_layers;
    const int vec = D.dtype == KVX_BF16 ? 8 : 4;   // elements per 16 bytes
    if (src->batch < 1) return bad(KVX_ERR_INVALID_ARG, "batch must be >= 1");
    if (src->max_seq < 0 || tgt->total_tokens < 0) return bad(KVX_ERR_INVALID_ARG, "negative size");
    if (!src->k || !src->v || !src->seq_len || !tgt->seq_off || !dst->k || !dst->v)
        return bad(KVX_ERR_INVALID_ARG, "NULL array");
    if ((tgt->span_lo == nullptr) != (tgt->span_hi == nullptr))
        return bad(KVX_ERR_INVALID_ARG, "span_lo and span_hi must both be set or both NULL");
    if (src->stride_s < D.src.head_dim || src->stride_h < 1 || src->stride_b < 1 || src->stride_s % vec ||
        src->stride_h % vec || src->stride_b % vec)
        return bad(KVX_ERR_INVALID_ARG, "source strides must be positive multiples of %d elements with "
                                        "stride_s >= head_dim", vec);
    if (!dst->paged) {
        if (dst->stride_t < D.dst.head_dim || dst->stride_h < 1 || dst->stride_b < 1 || dst->stride_t % vec ||
            dst->stride_h % vec || dst->stride_b % vec || dst->max_seq < 0)
            return bad(KVX_ERR_INVALID_ARG, "target strides must be positive multiples of %d elements with "
                                            "stride_t >= head_dim", vec);
    } else if (!dst->page_table || dst->page_size < 1 || dst->max_pages_per_seq < 1 || dst->num_pages < 1) {
        return bad(KVX_ERR_INVALID_ARG, "paged target needs page_table, page_size, max_pages_per_seq and "
                                        "num_pages >= 1");
    }
    memset(&P, 0, sizeof P);
    P.Hs = D.src.num_kv_heads; P.ds = D.src.head_dim;
    P.Ht = D.dst.num_kv_heads; P.dt = D.dst.head_dim;
    P.in_dim = g.in_dim; P.r = g.r; P.e = g.e; P.Lt = Lt;
    P.dense = g.dense; P.kl = g.kl; P.hpl = g.hpl;
    P.batch = src->batch; P.src_max_seq = src->max_seq;
    P.sb = src->stride_b; P.sh = src->stride_h; P.ss = src->stride_s;
    P.src_seq_len = src->seq_len; P.src_pos = src->pos;
    P.T_total = tgt->total_tokens; P.seq_off = tgt->seq_off;
    P.span_lo = tgt->span_lo; P.span_hi = tgt->span_hi; P.tgt_pos = tgt->pos;
    P.paged = dst->paged; P.dst_max_seq = dst->max_seq;
    P.db = dst->stride_b; P.dh = dst->stride_h; P.dts = dst->stride_t;
    P.page_table = dst->page_table; P.max_pages = dst->max_pages_per_seq;
    P.page_size = dst->page_size; P.num_pages = dst->num_pages;
    const int hs = D.src.head_dim / 2;
    P.rs = RopeTable{dev_turns, hs, D.src.rope_base > 0.0};
    P.rt = RopeTable{dev_turns + hs, D.dst.head_dim / 2, D.dst.rope_base > 0.0};
    P.rhalf_s = rope_rot_dim(D.src) / 2;
    P.rhalf_t = rope_rot_dim(D.dst) / 2;
    P.max_position = g.max_position;
    P.rope_same = g.rope_same;
    P.status = status;
    P.w = w;
    for (int i = 0; i < Lt * g.kl; ++i) {
        const int l = g.layer_map[i];
        P.src_k[i] = src->k[l]; P.src_v[i] = src->v[l];
        if (!P.src_k[i] || !P.src_v[i]) return bad(KVX_ERR_INVALID_ARG, "NULL cache pointer for source layer %d", l);
        if (!aligned16(P.src_k[i]) || !aligned16(P.src_v[i]))
            return bad(KVX_ERR_INVALID_ARG, "cache pointers must be 16-byte aligned (source layer %d)", l);
    }
    for (int j = 0; j < Lt; ++j) {
        P.dst_k[j] = dst->k[j]; P.dst_v[j] = dst->v[j];
        if (!P.dst_k[j] || !P.dst_v[j]) return bad(KVX_ERR_INVALID_ARG, "NULL cache pointer for target layer %d", j);
        if (!aligned16(P.dst_k[j]) || !aligned16(P.dst_v[j]))
            return bad(KVX_ERR_INVALID_ARG, "cache pointers must be 16-byte aligned (target layer %d)", j);
    }
    return KVX_OK;
}

}  // namespace kvx

extern "C" KVX_API kvx_status kvx_translator_create(const kvx_translator_desc* desc, const void* w_k,
                                                    const void* w_v, int32_t weights_on_device,
                                                    kvx_translator** out)
{
    if (!desc || !w_k || !w_v || !out) return fail(KVX_ERR_INVALID_ARG, "create: NULL argument");
    *out = nullptr;
    const kvx_model_geom& s = desc->src;
    const kvx_model_geom& d = desc->dst;
    char err[512];
    kvx_translator* t = new kvx_translator();
    kvx_status gst = make_geometry(desc, "create", t->geo, err);
    if (gst != KVX_OK) {
        delete t;
        g_last_error = err;
        return gst;
    }
    {
        const Geometry& g = t->geo;
        t->desc = g.desc;
        memcpy(t->layer_map, g.layer_map, sizeof t->layer_map);
        t->max_position = g.max_position;
        t->kl = g.kl; t->dense = g.dense; t->r = g.r; t->e = g.e; t->hpl = g.hpl; t->in_dim = g.in_dim;
        t->rope_same = g.rope_same;
    }

    if (cudaGetDevice(&t->device) != cudaSuccess ||
        cudaDeviceGetAttribute(&t->num_sms, cudaDevAttrMultiProcessorCount, t->device) != cudaSuccess) {
        delete t;
        return fail(KVX_ERR_CUDA, "create: no CUDA device");
    }

    // kernel choice
    t->tc = tc_config(t->in_dim, d.head_dim, s.head_dim, share_heads(t->dense, t->r, t->e, d.num_kv_heads));
    const bool tc_ok = desc->dtype == KVX_BF16 && t->tc.ok;
    if (desc->path == KVX_PATH_TCGEN05 && !tc_ok) {
        const int in_dim = t->in_dim;
        delete t;
        return fail(KVX_ERR_UNSUPPORTED, "create: no tcgen05 kernel for this geometry/dtype (in=%d, d_t=%d)",
                    in_dim, d.head_dim);
    }
    t->path = (desc->path == KVX_PATH_SIMT || !tc_ok) ? KVX_PATH_SIMT : KVX_PATH_TCGEN05;
    if (t->path == KVX_PATH_SIMT && simt_smem_bytes(t->in_dim, d.head_dim) > 200 * 1024) {
        delete t;
        return fail(KVX_ERR_UNSUPPORTED, "create: SIMT kernel shared memory too large");
    }

    const size_t elt = desc->dtype == KVX_BF16 ? 2 : 4;
    const size_t mat = (size_t)t->in_dim * d.head_dim;
    const size_t one = (size_t)d.num_layers * d.num_kv_heads * mat * elt;   // bytes of w_k
    kvx_status st = KVX_OK;
    void* raw = nullptr;
    cudaError_t ce;
    const cudaMemcpyKind kind = weights_on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;

    if (t->path == KVX_PATH_SIMT) {
        t->w_bytes = 2 * one;
        if (cudaMalloc(&t->w, t->w_bytes) != cudaSuccess) { st = fail(KVX_ERR_OOM, "create: weight allocation"); goto err; }
        if ((ce = cudaMemcpy(t->w, w_k, one, kind)) != cudaSuccess ||
            (ce = cudaMemcpy((char*)t->w + one, w_v, one, kind)) != cudaSuccess) {
            st = fail(KVX_ERR_CUDA, "create: weight copy: %s", cudaGetErrorString(ce));
            goto err;
        }
    } else {
        t->w_bytes = tc_weight_image_bytes(t->in_dim, d.head_dim, d.num_layers, d.num_kv_heads);
        if (cudaMalloc(&t->w, t->w_bytes) != cudaSuccess || cudaMalloc(&raw, 2 * one) != cudaSuccess) {
            st = fail(KVX_ERR_OOM, "create: weight allocation");
            goto err;
        }
        if ((ce = cudaMemcpy(raw, w_k, one, kind)) != cudaSuccess ||
            (ce = cudaMemcpy((char*)raw + one, w_v, one, kind)) != cudaSuccess ||
            (ce = launch_tc_weight_relayout(raw, (char*)raw + one, t->w, d.num_layers, d.num_kv_heads,
                                            t->in_dim, d.head_dim, t->tc.n_tile, rope_rot_dim(d) / 2, 0)) !=
                cudaSuccess ||
            (ce = cudaDeviceSynchronize()) != cudaSuccess) {
            st = fail(KVX_ERR_CUDA, "create: weight re-layout: %s", cudaGetErrorString(ce));
            goto err;
        }
        cudaFree(raw);
        raw = nullptr;
    }

    {   // rotation frequencies as fixed-point turns (kvx_common.cuh), from the geometry
        const int hs = s.head_dim / 2, hd = d.head_dim / 2;
        t->rope_bytes = (size_t)(hs + hd) * sizeof(unsigned long long);
        if (cudaMalloc(&t->rope, t->rope_bytes) != cudaSuccess) {
            st = fail(KVX_ERR_OOM, "create: table allocation");
            goto err;
        }
        memcpy(t->host_turns, t->geo.turns, sizeof t->host_turns);
        if ((ce = cudaMemcpy(t->rope, t->geo.turns, t->rope_bytes, cudaMemcpyHostToDevice)) != cudaSuccess) {
            st = fail(KVX_ERR_CUDA, "create: table upload: %s", cudaGetErrorString(ce));
            goto err;
        }
        t->rs = RopeTable{t->rope, hs, s.rope_base > 0.0};
        t->rt = RopeTable{t->rope + hs, hd, d.rope_base > 0.0};
    }
    if (cudaMalloc(&t->status, sizeof(unsigned)) != cudaSuccess) { st = fail(KVX_ERR_OOM, "create: status allocation"); goto err; }
    if (t->path == KVX_PATH_TCGEN05 && cudaMalloc(&t->plan, tc_plan_bytes(kvx_translator::kPlanTokens)) != cudaSuccess) {
        st = fail(KVX_ERR_OOM, "create: span plan allocation");
        goto err;
    }
    if ((ce = cudaMemset(t->status, 0, sizeof(unsigned))) != cudaSuccess ||
        (ce = cudaDeviceSynchronize()) != cudaSuccess) {
        st = fail(KVX_ERR_CUDA, "create: %s", cudaGetErrorString(ce));
        goto err;
    }
    *out = t;
    return KVX_OK;
err:
    if (raw) cudaFree(raw);
    free_translator(t);
    return st;
}

extern "C" KVX_API kvx_status kvx_translator_create_low_rank(const kvx_translator_desc* desc, int32_t rank,
                                                             const void* a_k, const void* b_k, const void* a_v,
                                                             const void* b_v, int32_t weights_on_device,
                                                             kvx_translator** out)
{
    if (!desc || !a_k || !b_k || !a_v || !b_v || !out) return fail(KVX_ERR_INVALID_ARG, "create_low_rank: NULL argument");
    *out = nullptr;
    if (rank < 1 || rank > 1024) return fail(KVX_ERR_INVALID_ARG, "create_low_rank: rank %d outside [1, 1024]", rank);
    const kvx_model_geom& s = desc->src;
    const kvx_model_geom& d = desc->dst;
    if (s.num_layers < 1 || d.num_layers < 1 || s.num_kv_heads < 1 || d.num_kv_heads < 1 ||
        d.num_layers > KVX_MAX_TARGET_LAYERS || !head_dim_ok(s.head_dim) || !head_dim_ok(d.head_dim))
        return fail(KVX_ERR_INVALID_ARG, "create_low_rank: bad layer, head or head_dim counts");
    if (s.num_kv_heads % d.num_kv_heads != 0 && d.num_kv_heads % s.num_kv_heads != 0)
        return fail(KVX_ERR_UNSUPPORTED, "create_low_rank: neither KV head count divides the other");
    if (desc->dtype != KVX_BF16 && desc->dtype != KVX_FP32)
        return fail(KVX_ERR_INVALID_ARG, "create_low_rank: unknown dtype %d", desc->dtype);
    // the input width, as kvx_translator_create derives it (it validates the rest)
    const int kl = desc->layers_per_target > 1 ? desc->layers_per_target : 1;
    const int hpl = desc->form == KVX_FORM_DENSE ? s.num_kv_heads
                                                 : (s.num_kv_heads >= d.num_kv_heads ? s.num_kv_heads / d.num_kv_heads : 1);
    const long long in_dim = (long long)kl * hpl * s.head_dim;
    if (in_dim > 1024) return fail(KVX_ERR_UNSUPPORTED, "create_low_rank: translator input width %lld > 1024", in_dim);
    const size_t elt = desc->dtype == KVX_BF16 ? 2 : 4;
    const int n = d.num_layers * d.num_kv_heads;
    const size_t a_bytes = (size_t)n * in_dim * rank * elt, b_bytes = (size_t)n * rank * d.head_dim * elt;
    const size_t w_bytes = (size_t)n * in_dim * d.head_dim * elt;
    char* buf = nullptr;
    if (cudaMalloc(&buf, 2 * (a_bytes + b_bytes + w_bytes)) != cudaSuccess)
        return fail(KVX_ERR_OOM, "create_low_rank: factor allocation");
    char *ak = buf, *av = ak + a_bytes, *bk = av + a_bytes, *bv = bk + b_bytes, *wk = bv + b_bytes, *wv = wk + w_bytes;
    const cudaMemcpyKind kind = weights_on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
    cudaError_t ce;
    if ((ce = cudaMemcpy(ak, a_k, a_bytes, kind)) != cudaSuccess || (ce = cudaMemcpy(av, a_v, a_bytes, kind)) != cudaSuccess ||
        (ce = cudaMemcpy(bk, b_k, b_bytes, kind)) != cudaSuccess || (ce = cudaMemcpy(bv, b_v, b_bytes, kind)) != cudaSuccess ||
        (ce = launch_fold_low_rank(ak, bk, wk, n, (int)in_dim, rank, d.head_dim, desc->dtype, 0)) != cudaSuccess ||
        (ce = launch_fold_low_rank(av, bv, wv, n, (int)in_dim, rank, d.head_dim, desc->dtype, 0)) != cudaSuccess ||
        (ce = cudaDeviceSynchronize()) != cudaSuccess) {
        cudaFree(buf);
        return fail(KVX_ERR_CUDA, "create_low_rank: factor product: %s", cudaGetErrorString(ce));
    }
    const kvx_status st = kvx_translator_create(desc, wk, wv, 1, out);
    cudaFree(buf);
    return st;
}

// The translation launch(es) of kvx_translate; plain_stores: the kernels write the target rows
// with thread stores (a destination on another device).
static kvx_status translate_impl(kvx_translator* tr, const kvx_src_kv* src, const kvx_tgt_tokens* tgt,
                                 const kvx_dst_kv* dst, void* stream, int plain_stores)
{
    if (!tr || !src || !tgt || !dst) return fail(KVX_ERR_INVALID_ARG, "translate: NULL argument");
    const kvx_translator_desc& D = tr->desc;
    const int Lt = D.dst.num_layers;
    tr->last_launches = 0;
    tr->last_span_tokens = 0;
    TranslateParams P;
    char err[512];
    const kvx_status pst = make_params(tr->geo, tr->rope, tr->status, tr->w, src, tgt, dst, P, "translate", err);
    if (pst != KVX_OK) {
        g_last_error = err;
        return pst;
    }
    P.wait_ns = tr->dbg_wait_ns;
    P.stall_unit1 = tr->dbg_stall_unit1;
    tr->dbg_wait_ns = 0;
    tr->dbg_stall_unit1 = 0;
    if (tgt->total_tokens == 0) return KVX_OK;
    P.plain_stores = plain_stores;
    cudaError_t ce;
    // partial rotary heads (rotary_dim < head_dim on either side) take the span kernel, which
    // pairs channels at rotary_dim/2; the identity kernel pairs whole heads
    const bool whole_head_rope = rope_rot_dim(D.src) == D.src.head_dim && rope_rot_dim(D.dst) == D.dst.head_dim;
    if (tr->path == KVX_PATH_TCGEN05 && !tgt->span_lo && whole_head_rope &&
        aligned_supported(tr->in_dim, D.dst.head_dim, D.src.head_dim, share_heads(tr->dense, tr->r, tr->e, D.dst.num_kv_heads),
                          Lt, src->batch, tr->kl)) {
        // identity alignment: tensor-TMA fed kernel
        if (tr->maps.empty()) tr->maps.resize((size_t)2 * KVX_MAX_ALIGNED_LAYERS * kvx_translator::kMapWays);
        const void* maps[2 * KVX_MAX_ALIGNED_LAYERS];
        for (int j = 0; j < Lt; ++j)
            for (int kv = 0; kv < 2; ++kv) {
                maps[2 * j + kv] = source_map(tr, j, kv, kv ? P.src_v[j] : P.src_k[j], src);
                if (!maps[2 * j + kv])
                    return fail(KVX_ERR_INVALID_ARG, "translate: cannot describe the source cache of layer %d to the "
                                                     "tensor-copy unit (strides, sizes)", tr->layer_map[j]);
            }
        ce = launch_translate_tc_aligned(P, maps, tr->host_turns, tr->num_sms, (cudaStream_t)stream);
        tr->last_launches = 1;
    } else if (tr->path == KVX_PATH_TCGEN05) {
        ce = launch_translate_tc(P, tr->tc, tr->num_sms, tr->plan, kvx_translator::kPlanTokens, (cudaStream_t)stream,
                                 &tr->last_launches);
        tr->last_span_tokens = P.T_total;
    } else {
        ce = launch_translate_simt(P, D.dtype, (cudaStream_t)stream);
        tr->last_launches = 1;
    }
    if (ce != cudaSuccess) return fail(KVX_ERR_CUDA, "translate: launch failed: %s", cudaGetErrorString(ce));
    return KVX_OK;
}

extern "C" KVX_API kvx_status kvx_translate(kvx_translator* tr, const kvx_src_kv* src, const kvx_tgt_tokens* tgt,
                                            const kvx_dst_kv* dst, void* stream)
{
    return translate_impl(tr, src, tgt, dst, stream, 0);
}

// ---------------------------------------------------------------------------------------------
// Writing the translated cache into the target model's GPU (the handoff's peer copy).
static std::mutex g_peer_mutex;
static unsigned long long g_peer_enabled[64];   // [device] bit p: peer access to device p enabled by kvx_enable_peer

extern "C" KVX_API kvx_status kvx_enable_peer(int32_t peer_device)
{
    int cur = 0, n = 0;
    CUDA_OR_FAIL(cudaGetDevice(&cur));
    CUDA_OR_FAIL(cudaGetDeviceCount(&n));
    if (peer_device < 0 || peer_device >= n || peer_device >= 64 || cur >= 64)
        return fail(KVX_ERR_INVALID_ARG, "enable_peer: no device %d", peer_device);
    if (peer_device == cur) return KVX_OK;
    std::lock_guard<std::mutex> lock(g_peer_mutex);
    if (g_peer_enabled[cur] >> peer_device & 1ull) return KVX_OK;
    int can = 0;
    CUDA_OR_FAIL(cudaDeviceCanAccessPeer(&can, cur, peer_device));
    if (!can) return fail(KVX_ERR_UNSUPPORTED, "enable_peer: device %d cannot access device %d", cur, peer_device);
    cudaError_t e = cudaDeviceEnablePeerAccess(peer_device, 0);
    if (e == cudaErrorPeerAccessAlreadyEnabled) {
        cudaGetLastError();   // already enabled by the caller: not an error here
        e = cudaSuccess;
    }
    if (e != cudaSuccess) return fail(KVX_ERR_CUDA, "enable_peer: %s", cudaGetErrorString(e));
    g_peer_enabled[cur] |= 1ull << peer_device;
    return KVX_OK;
}

// Device of a caller pointer (-1 if it is not device memory).
static int pointer_device(const void* p)
{
    cudaPointerAttributes a{};
    if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
        cudaGetLastError();
        return -1;
    }
    return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged ? a.device : -1;
}

extern "C" KVX_API kvx_status kvx_translate_to_device(kvx_translator* tr, const kvx_src_kv* src,
                                                      const kvx_tgt_tokens* tgt, const kvx_dst_kv* dst,
                                                      int32_t dst_device, int32_t mode, const kvx_dst_kv* staging,
                                                      void* stream)
{
    if (!tr || !src || !tgt || !dst) return fail(KVX_ERR_INVALID_ARG, "translate_to_device: NULL argument");
    int cur = 0;
    CUDA_OR_FAIL(cudaGetDevice(&cur));
    const int Lt = tr->desc.dst.num_layers;
    if (!dst->k || !dst->v) return fail(KVX_ERR_INVALID_ARG, "translate_to_device: NULL array");
    for (int j = 0; j < Lt; ++j)
        for (const void* p : {(const void*)dst->k[j], (const void*)dst->v[j]})
            if (p && pointer_device(p) != dst_device)
                return fail(KVX_ERR_INVALID_ARG, "translate_to_device: target layer %d is not memory of device %d",
                            j, dst_device);
    if (mode == KVX_PEER_STORES) {
        if (dst_device != cur) {
            std::lock_guard<std::mutex> lock(g_peer_mutex);
            if (cur >= 64 || dst_device < 0 || dst_device >= 64 || !(g_peer_enabled[cur] >> dst_device & 1ull))
                return fail(KVX_ERR_INVALID_ARG, "translate_to_device: call kvx_enable_peer(%d) on device %d first",
                            dst_device, cur);
        }
        return translate_impl(tr, src, tgt, dst, stream, 1);
    }
    if (mode != KVX_PEER_STAGED) return fail(KVX_ERR_INVALID_ARG, "translate_to_device: unknown mode %d", mode);
    if (!staging || !staging->k || !staging->v)
        return fail(KVX_ERR_INVALID_ARG, "translate_to_device: the staged mode needs a staging cache");
    if (dst->paged || staging->paged)
        return fail(KVX_ERR_UNSUPPORTED, "translate_to_device: the staged mode copies whole contiguous caches; "
                                         "write paged pools with KVX_PEER_STORES");
    if (staging->stride_b != dst->stride_b || staging->stride_h != dst->stride_h ||
        staging->stride_t != dst->stride_t || staging->max_seq != dst->max_seq)
        return fail(KVX_ERR_INVALID_ARG, "translate_to_device: staging and target caches differ in layout");
    for (int j = 0; j < Lt; ++j)
        for (const void* p : {(const void*)staging->k[j], (const void*)staging->v[j]})
            if (p && pointer_device(p) != cur)
                return fail(KVX_ERR_INVALID_ARG, "translate_to_device: staging layer %d is not memory of device %d",
                            j, cur);
    const kvx_status st = translate_impl(tr, src, tgt, staging, stream, 0);
    if (st != KVX_OK || tgt->total_tokens == 0) return st;
    // every staged tensor, whole: [batch][heads][max_seq][head_dim] under the strides
    const size_t elt = tr->desc.dtype == KVX_BF16 ? 2 : 4;
    const int64_t extent = (int64_t)(src->batch - 1) * dst->stride_b + (int64_t)(tr->desc.dst.num_kv_heads - 1) * dst->stride_h +
                           (int64_t)(dst->max_seq > 0 ? dst->max_seq - 1 : 0) * dst->stride_t + tr->desc.dst.head_dim;
    for (int j = 0; j < Lt; ++j)
        for (int kv = 0; kv < 2; ++kv) {
            void* to = kv ? dst->v[j] : dst->k[j];
            const void* from = kv ? staging->v[j] : staging->k[j];
            CUDA_OR_FAIL(cudaMemcpyPeerAsync(to, dst_device, from, cur, (size_t)extent * elt, (cudaStream_t)stream));
        }
    return KVX_OK;
}

extern "C" KVX_API kvx_status kvx_build_alignment(int32_t batch, int32_t total_src, int32_t total_tgt,
                                                  const int32_t* src_seq_off, const int32_t* src_end,
                                                  const int32_t* tgt_seq_off, const int32_t* tgt_end,
                                                  int32_t* span_lo, int32_t* span_hi, uint32_t* dev_status,
                                                  void* stream)
{
    if (batch < 1 || total_src < 0 || total_tgt < 0)
        return fail(KVX_ERR_INVALID_ARG, "build_alignment: bad sizes");
    if (total_tgt == 0) return KVX_OK;
    if (!src_seq_off || !tgt_seq_off || !tgt_end || !span_lo || !span_hi || (total_src > 0 && !src_end))
        return fail(KVX_ERR_INVALID_ARG, "build_alignment: NULL array");
    cudaError_t ce = launch_build_alignment(batch, total_tgt, src_seq_off, src_end, tgt_seq_off, tgt_end, span_lo,
                                            span_hi, dev_status, (cudaStream_t)stream);
    if (ce != cudaSuccess) return fail(KVX_ERR_CUDA, "build_alignment: %s", cudaGetErrorString(ce));
    return KVX_OK;
}

extern "C" KVX_API kvx_status kvx_get_device_status(kvx_translator* tr, void* stream, uint32_t* bits, int32_t clear)
{
    if (!tr) return fail(KVX_ERR_INVALID_ARG, "get_device_status: NULL translator");
    unsigned v = 0;
    CUDA_OR_FAIL(cudaStreamSynchronize((cudaStream_t)stream));
    CUDA_OR_FAIL(cudaMemcpy(&v, tr->status, sizeof v, cudaMemcpyDeviceToHost));
    if (clear) CUDA_OR_FAIL(cudaMemset(tr->status, 0, sizeof v));
    if (bits) *bits = v;
    if (v) return fail(KVX_ERR_DEVICE_STATUS, "device status 0x%x", v);
    return KVX_OK;
}

extern "C" KVX_API kvx_status kvx_get_info(const kvx_translator* tr, kvx_translator_info* info)
{
    if (!tr || !info) return fail(KVX_ERR_INVALID_ARG, "get_info: NULL argument");
    info->path = tr->path;
    info->group_in = tr->in_dim;
    info->n_tile = tr->path == KVX_PATH_TCGEN05 ? tr->tc.n_tile : 0;
    info->smem_bytes = tr->path == KVX_PATH_TCGEN05 ? tr->tc.smem_bytes
                                                    : (int)simt_smem_bytes(tr->in_dim, tr->desc.dst.head_dim);
    info->threads = tr->path == KVX_PATH_TCGEN05 ? tr->tc.threads : 256;
    info->num_sms = tr->num_sms;
    info->weight_bytes = (int64_t)tr->w_bytes;
    info->table_bytes = (int64_t)tr->rope_bytes;
    return KVX_OK;
}

extern "C" KVX_API int32_t kvx_launches_per_translate(const kvx_translator* tr) { return tr ? tr->last_launches : 0; }

extern "C" KVX_API kvx_status kvx_debug_stall_next_translate(kvx_translator* tr, int32_t unit, int32_t wait_us)
{
    if (!tr || unit < 0 || wait_us < 1 || wait_us > 1000000)
        return fail(KVX_ERR_INVALID_ARG, "debug_stall_next_translate: bad arguments");
    tr->dbg_stall_unit1 = unit + 1;
    tr->dbg_wait_ns = (unsigned long long)wait_us * 1000ull;
    return KVX_OK;
}

extern "C" KVX_API kvx_status kvx_span_plan_stats(kvx_translator* tr, void* stream, int64_t* counts)
{
    if (!tr || !counts) return fail(KVX_ERR_INVALID_ARG, "span_plan_stats: NULL argument");
    if (tr->last_span_tokens <= 0 || !tr->plan)
        return fail(KVX_ERR_INVALID_ARG, "span_plan_stats: the last kvx_translate did not run the span kernel");
    int nsub = 0, ent_off = 0;
    tc_plan_layout(tr->last_span_tokens, kvx_translator::kPlanTokens, &nsub, &ent_off);
    std::vector<int4> ent((size_t)nsub * 32);
    CUDA_OR_FAIL(cudaStreamSynchronize((cudaStream_t)stream));
    CUDA_OR_FAIL(cudaMemcpy(ent.data(), (const int4*)tr->plan + ent_off, ent.size() * sizeof(int4),
                            cudaMemcpyDeviceToHost));
    int64_t staged = 0, global = 0, subs_global = 0;
    for (int sub = 0; sub < nsub; ++sub) {
        bool any = false;
        for (int i = 0; i < 32; ++i) {
            const int4 e = ent[(size_t)sub * 32 + i];
            if (((unsigned)e.x >> 16) >= 32u) continue;          // token past the end
            if ((short)(e.x & 0xFFFF) < 0) { ++global; any = true; }
            else ++staged;
        }
        subs_global += any;
    }
    counts[0] = nsub;
    counts[1] = staged;
    counts[2] = global;
    counts[3] = subs_global;
    return KVX_OK;
}

extern "C" KVX_API kvx_status kvx_destroy(kvx_translator* tr)
{
    if (!tr) return KVX_OK;
    cudaDeviceSynchronize();
    free_translator(tr);
    return KVX_OK;
}
