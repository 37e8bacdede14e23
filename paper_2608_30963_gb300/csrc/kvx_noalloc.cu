// kvx_noalloc.cu -- kvx_translate_static: translation without any device allocation.
//
// kvx_translator_create allocates device memory for its copy of the weights,
// the rotation frequencies and a status word.  Some callers cannot do that at
// translation time: a serving process whose device memory belongs to a caching
// allocator that forbids raw cudaMalloc, a runtime with a fixed memory budget
// reserved at start-up, or code on a latency-critical path where cudaMalloc /
// cudaFree would synchronise the device.  For them this entry point runs the
// CUDA-core translation kernel with all of its scratch in one file-scope
// device array that exists for as long as the library is loaded.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <mutex>

#include "kvx_common.cuh"
#include "kvx_kernels.h"

namespace kvx {
namespace {

// Scratch layout: [status word, 256 B][source turns][target turns][weights K | V].
constexpr size_t kStatusBytes = 256;
constexpr size_t kTurnsBytes = 2 * 128 * sizeof(unsigned long long);   // two models, d/2 <= 128
constexpr size_t kWeightsOffset = kStatusBytes + kTurnsBytes;

__device__ __align__(256) unsigned char g_static_scratch[KVX_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
// Device address of g_static_scratch per device, and the context it was looked up in: the
// address belongs to that context, so a call under another context (a non-primary one, or the
// primary context re-created after cudaDeviceReset) looks it up again.
unsigned char* g_scratch_addr[kMaxDevices];
void* g_scratch_ctx[kMaxDevices];

// The calling thread's current driver context (NULL if it cannot be read).
void* current_context()
{
    using GetCurrent = int (*)(void**);
    static GetCurrent fn = [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            p = nullptr;
        return (GetCurrent)p;
    }();
    void* ctx = nullptr;
    if (!fn || fn(&ctx) != 0) return nullptr;
    return ctx;
}

thread_local char g_msg[512];

kvx_status fail(kvx_status s, const char* fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_msg, sizeof g_msg, fmt, ap);
    va_end(ap);
    return s;
}

// Fixed-point rotation turns 2^64 f_i / 2 pi (in double, truncated to an integer, as on the
// host), f_i the model's scheduled frequency of pair i (0 for the pairs of a partial rotary
// head that do not rotate), written on the device.
__global__ void static_turns_kernel(unsigned long long* out, const kvx_model_geom g)
{
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= g.head_dim / 2) return;
    if (g.rope_base <= 0.0 || i >= rope_rot_dim(g) / 2) { out[i] = 0ull; return; }
    out[i] = (unsigned long long)ldexp(rope_inv_freq(g, i) / (2.0 * 3.14159265358979323846), 64);
}

}  // namespace
}  // namespace kvx

using namespace kvx;

extern "C" KVX_API const char* kvx_static_last_error(void) { return g_msg; }

extern "C" KVX_API kvx_status kvx_translate_static(const kvx_translator_desc* desc, const void* w_k, const void* w_v,
                                                   const kvx_src_kv* src, const kvx_tgt_tokens* tgt,
                                                   const kvx_dst_kv* dst, uint32_t* status_bits, void* stream)
{
    g_msg[0] = 0;
    if (!desc || !w_k || !w_v || !src || !tgt || !dst) return fail(KVX_ERR_INVALID_ARG, "translate_static: NULL argument");
    const kvx_model_geom& s = desc->src;
    const kvx_model_geom& d = desc->dst;
    auto hd_ok = [](int h) { return h == 64 || h == 128 || h == 256; };
    if (s.num_layers < 1 || d.num_layers < 1 || s.num_kv_heads < 1 || d.num_kv_heads < 1)
        return fail(KVX_ERR_INVALID_ARG, "translate_static: layer and head counts must be >= 1");
    if (d.num_layers > KVX_MAX_TARGET_LAYERS)
        return fail(KVX_ERR_UNSUPPORTED, "translate_static: at most %d target layers", KVX_MAX_TARGET_LAYERS);
    if (!hd_ok(s.head_dim) || !hd_ok(d.head_dim))
        return fail(KVX_ERR_UNSUPPORTED, "translate_static: head dims must be 64, 128 or 256");
    if (s.num_kv_heads % d.num_kv_heads != 0 && d.num_kv_heads % s.num_kv_heads != 0)
        return fail(KVX_ERR_UNSUPPORTED, "translate_static: neither KV head count divides the other");
    if (desc->dtype != KVX_BF16 && desc->dtype != KVX_FP32)
        return fail(KVX_ERR_INVALID_ARG, "translate_static: unknown dtype %d", desc->dtype);
    if (desc->form != KVX_FORM_GROUPED || desc->layers_per_target > 1)
        return fail(KVX_ERR_UNSUPPORTED, "translate_static: only the per-KV-head form over one source layer per "
                                         "target layer");
    if (!rope_schedule_ok(s) || !rope_schedule_ok(d))
        return fail(KVX_ERR_INVALID_ARG, "translate_static: unknown rope_type or schedule parameters out of range");
    const int max_pos = desc->max_position ? desc->max_position : (1 << 24);
    if (max_pos < 1 || max_pos > (1 << 30))
        return fail(KVX_ERR_INVALID_ARG, "translate_static: max_position must be in [1, 1<<30]");
    const int r = s.num_kv_heads >= d.num_kv_heads ? s.num_kv_heads / d.num_kv_heads : 1;
    const int e = s.num_kv_heads >= d.num_kv_heads ? 1 : d.num_kv_heads / s.num_kv_heads;
    const int in_dim = s.num_kv_heads >= d.num_kv_heads ? r * s.head_dim : s.head_dim;
    if (in_dim > 512 || simt_smem_bytes(in_dim, d.head_dim) > 200 * 1024)
        return fail(KVX_ERR_UNSUPPORTED, "translate_static: translator input width %d too large", in_dim);
    int layer_map[KVX_MAX_TARGET_LAYERS];
    for (int j = 0; j < d.num_layers; ++j) {
        if (desc->layer_map) {
            if (desc->layer_map[j] < 0 || desc->layer_map[j] >= s.num_layers)
                return fail(KVX_ERR_INVALID_ARG, "translate_static: layer_map[%d] out of range", j);
            layer_map[j] = desc->layer_map[j];
        } else {
            layer_map[j] = d.num_layers == 1 ? 0
                                             : (int)((2LL * j * (s.num_layers - 1) + (d.num_layers - 1)) /
                                                     (2LL * (d.num_layers - 1)));
        }
    }
    const size_t elt = desc->dtype == KVX_BF16 ? 2 : 4;
    const size_t one = (size_t)d.num_layers * d.num_kv_heads * in_dim * d.head_dim * elt;
    if (kWeightsOffset + 2 * one > (size_t)KVX_STATIC_SCRATCH_BYTES)
        return fail(KVX_ERR_UNSUPPORTED, "translate_static: weights need %zu bytes, the static scratch holds %zu",
                    2 * one, (size_t)KVX_STATIC_SCRATCH_BYTES - kWeightsOffset);

    // argument checks shared with kvx_translate
    const int vec = desc->dtype == KVX_BF16 ? 8 : 4;
    if (src->batch < 1 || src->max_seq < 0 || tgt->total_tokens < 0)
        return fail(KVX_ERR_INVALID_ARG, "translate_static: bad sizes");
    if (!src->k || !src->v || !src->seq_len || !tgt->seq_off || !dst->k || !dst->v)
        return fail(KVX_ERR_INVALID_ARG, "translate_static: NULL array");
    if ((tgt->span_lo == nullptr) != (tgt->span_hi == nullptr))
        return fail(KVX_ERR_INVALID_ARG, "translate_static: span_lo and span_hi must both be set or both NULL");
    if (src->stride_s < s.head_dim || src->stride_h < 1 || src->stride_b < 1 || src->stride_s % vec ||
        src->stride_h % vec || src->stride_b % vec)
        return fail(KVX_ERR_INVALID_ARG, "translate_static: bad source strides");
    if (!dst->paged) {
        if (dst->stride_t < d.head_dim || dst->stride_h < 1 || dst->stride_b < 1 || dst->stride_t % vec ||
            dst->stride_h % vec || dst->stride_b % vec || dst->max_seq < 0)
            return fail(KVX_ERR_INVALID_ARG, "translate_static: bad target strides");
    } else if (!dst->page_table || dst->page_size < 1 || dst->max_pages_per_seq < 1 || dst->num_pages < 1) {
        return fail(KVX_ERR_INVALID_ARG, "translate_static: bad page table");
    }

    // once per device, with that device current: the device address of the scratch array
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return fail(KVX_ERR_CUDA, "translate_static: no usable current device");
    unsigned char* scratch = nullptr;
    {
        std::lock_guard<std::mutex> lock(g_setup_mutex);
        void* ctx = current_context();
        if (!g_scratch_addr[dev] || ctx != g_scratch_ctx[dev]) {
            void* ptr = nullptr;
            const cudaError_t ce = cudaGetSymbolAddress(&ptr, g_static_scratch);
            if (ce != cudaSuccess || !ptr)
                return fail(KVX_ERR_CUDA, "translate_static: cudaGetSymbolAddress: %s", cudaGetErrorString(ce));
            g_scratch_addr[dev] = (unsigned char*)ptr;
            g_scratch_ctx[dev] = current_context();   // the lookup made the runtime's context current
        }
        scratch = g_scratch_addr[dev];
    }
    cudaStream_t st = (cudaStream_t)stream;
    unsigned* status = (unsigned*)scratch;
    unsigned long long* turns = (unsigned long long*)(scratch + kStatusBytes);
    unsigned char* wts = scratch + kWeightsOffset;
    cudaError_t ce;
    if ((ce = cudaMemsetAsync(status, 0, sizeof(unsigned), st)) != cudaSuccess ||
        (ce = cudaMemcpyAsync(wts, w_k, one, cudaMemcpyDeviceToDevice, st)) != cudaSuccess ||
        (ce = cudaMemcpyAsync(wts + one, w_v, one, cudaMemcpyDeviceToDevice, st)) != cudaSuccess)
        return fail(KVX_ERR_CUDA, "translate_static: %s", cudaGetErrorString(ce));
    static_turns_kernel<<<1, 128, 0, st>>>(turns, s);
    static_turns_kernel<<<1, 128, 0, st>>>(turns + 128, d);
    if ((ce = cudaGetLastError()) != cudaSuccess)
        return fail(KVX_ERR_CUDA, "translate_static: %s", cudaGetErrorString(ce));

    if (tgt->total_tokens > 0) {
        TranslateParams P;
        memset(&P, 0, sizeof P);
        P.Hs = s.num_kv_heads; P.ds = s.head_dim; P.Ht = d.num_kv_heads; P.dt = d.head_dim;
        P.in_dim = in_dim; P.r = r; P.e = e; P.Lt = d.num_layers;
        P.dense = 0; P.kl = 1; P.hpl = r;
        P.batch = src->batch; P.src_max_seq = src->max_seq;
        P.sb = src->stride_b; P.sh = src->stride_h; P.ss = src->stride_s;
        P.src_seq_len = src->seq_len; P.src_pos = src->pos;
        P.T_total = tgt->total_tokens; P.seq_off = tgt->seq_off;
        P.span_lo = tgt->span_lo; P.span_hi = tgt->span_hi; P.tgt_pos = tgt->pos;
        P.paged = dst->paged; P.dst_max_seq = dst->max_seq;
        P.db = dst->stride_b; P.dh = dst->stride_h; P.dts = dst->stride_t;
        P.page_table = dst->page_table; P.max_pages = dst->max_pages_per_seq;
        P.page_size = dst->page_size; P.num_pages = dst->num_pages;
        P.rs = RopeTable{turns, s.head_dim / 2, s.rope_base > 0.0};
        P.rt = RopeTable{turns + 128, d.head_dim / 2, d.rope_base > 0.0};
        P.rhalf_s = rope_rot_dim(s) / 2;
        P.rhalf_t = rope_rot_dim(d) / 2;
        P.max_position = max_pos;
        P.status = status;
        P.w = wts;
        for (int j = 0; j < d.num_layers; ++j) {
            P.src_k[j] = src->k[layer_map[j]]; P.src_v[j] = src->v[layer_map[j]];
            P.dst_k[j] = dst->k[j]; P.dst_v[j] = dst->v[j];
            if (!P.src_k[j] || !P.src_v[j] || !P.dst_k[j] || !P.dst_v[j])
                return fail(KVX_ERR_INVALID_ARG, "translate_static: NULL cache pointer for target layer %d", j);
        }
        if ((ce = launch_translate_simt(P, desc->dtype, st)) != cudaSuccess)
            return fail(KVX_ERR_CUDA, "translate_static: launch failed: %s", cudaGetErrorString(ce));
    }
    if (status_bits) {
        unsigned v = 0;
        if ((ce = cudaMemcpyAsync(&v, status, sizeof v, cudaMemcpyDeviceToHost, st)) != cudaSuccess ||
            (ce = cudaStreamSynchronize(st)) != cudaSuccess)
            return fail(KVX_ERR_CUDA, "translate_static: %s", cudaGetErrorString(ce));
        *status_bits = v;
        if (v) return fail(KVX_ERR_DEVICE_STATUS, "translate_static: device status 0x%x", v);
    }
    return KVX_OK;
}
