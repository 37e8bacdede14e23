/*
 * kvx.h -- C ABI of the cross-model KV translation library (libkvx.so).
 *
 * Cross-model KV sharing (paper Section 4) turns the KV cache a source model A
 * built for a context C into a cache a different target model B can decode
 * from without its own prefill:  KV^_B(C) = T_{A->B}(KV_A(C)).  Section 5
 * writes the translator as a parameterised map T_theta and lists the
 * granularities it may act on (layers, groups of layers, KV heads, ...).  This
 * library implements a per-target-layer, per-target-KV-head linear T_theta:
 *
 *   for target layer j, target KV head h, target token t (span [lo_t, hi_t)):
 *     K^_j,h[t] = R_dst(p_t) . W_K[j,h]^T . mean_{s in span} concat_g R_src(-p_s) K_{map[j],g}[s]
 *     V^_j,h[t] =              W_V[j,h]^T . mean_{s in span} concat_g            V_{map[j],g}[s]
 *
 * where map[] is the layer alignment, g runs over the source KV heads grouped
 * into target head h (GQA regrouping), R(p) is the half-split rotary map at
 * position p (angle p * base^(-2i/d) on channel pair (i, i+d/2)), and the
 * result is written into the target model's contiguous or paged KV cache
 * (the paper's "cache assembly", Section 6.1 and Table 4).
 *
 * Conventions for every entry point:
 *   - All sizes are element counts unless a name says bytes.
 *   - "device" pointers are CUDA device (or managed) memory of the current
 *     device; "host" pointers are ordinary host memory.  The caller owns every
 *     buffer it passes; the library never frees a caller buffer.
 *   - stream is a cudaStream_t passed as void* (NULL = legacy default stream).
 *   - Calls return a kvx_status; on failure kvx_last_error() gives a message
 *     for the calling thread.  Argument errors are detected on the host before
 *     anything is launched.  Data errors that only the device can see (a span,
 *     position or page index out of range) are clamped or skipped on the
 *     device and recorded in the translator's device status word; read it with
 *     kvx_get_device_status().  No kernel traps or waits without bound.
 */
#ifndef KVX_H
#define KVX_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define KVX_API __attribute__((visibility("default")))

typedef enum {
    KVX_OK = 0,
    KVX_ERR_INVALID_ARG = 1,    /* a pointer, size or stride is invalid */
    KVX_ERR_UNSUPPORTED = 2,    /* a geometry the library has no kernel for */
    KVX_ERR_CUDA = 3,           /* a CUDA runtime call failed */
    KVX_ERR_OOM = 4,            /* device allocation failed (create only) */
    KVX_ERR_DEVICE_STATUS = 5   /* kvx_get_device_status found a nonzero status */
} kvx_status;

typedef enum {
    KVX_BF16 = 0,               /* bfloat16 caches and weights; fp32 arithmetic */
    KVX_FP32 = 1                /* float32 caches and weights; fp32 arithmetic */
} kvx_dtype;

typedef enum {
    KVX_PATH_AUTO = 0,          /* tcgen05 kernel for bf16 where supported, else SIMT */
    KVX_PATH_SIMT = 1,          /* CUDA-core kernel (any supported geometry, both dtypes) */
    KVX_PATH_TCGEN05 = 2        /* tensor-core kernel (bf16 only) */
} kvx_path;

/* Bits of the device status word. */
#define KVX_DEV_SPAN_CLAMPED  0x01u  /* a span fell outside [0, seq_len) or was empty; clamped */
#define KVX_DEV_POS_CLAMPED   0x02u  /* a RoPE position fell outside [0, max_position); clamped */
#define KVX_DEV_PAGE_INVALID  0x04u  /* a page-table entry fell outside [0, num_pages); row not written */
#define KVX_DEV_SEQ_CLAMPED   0x08u  /* a seq_len exceeded max_seq, or a target row fell outside the cache */
#define KVX_DEV_WAIT_TIMEOUT  0x10u  /* an on-chip pipeline wait gave up after ~1 s; output incomplete */

#define KVX_MAX_TARGET_LAYERS 128  /* target layers a translator may have */

/* Frequency schedule of a model's rotary encoding.  The plain schedule rotates channel pair
 * (i, i+d/2) by p * f_i with f_i = base^(-2i/d).  The paper names the model pairs it evaluates
 * (Section 6.1) but not their position encodings; these schedules are the ones the named
 * families publish (Llama-3.1 ships the LLAMA3 schedule). */
typedef enum {
    KVX_ROPE_DEFAULT = 0,       /* f_i = base^(-2i/d) */
    KVX_ROPE_LINEAR = 1,        /* position interpolation: angle (p / factor) * f_i */
    KVX_ROPE_LLAMA3 = 2         /* frequency-dependent: with wavelength w_i = 2 pi / f_i,
                                   lo_w = original_max_position / low_freq_factor and
                                   hi_w = original_max_position / high_freq_factor,
                                   f_i is kept where w_i < hi_w, divided by factor where
                                   w_i > lo_w, and in between blended as
                                   (1 - m) f_i / factor + m f_i with
                                   m = (original_max_position / w_i - low_freq_factor) /
                                       (high_freq_factor - low_freq_factor) */
} kvx_rope_type;

/* Geometry of one model's KV cache.  A zero-initialised tail (rope_type 0) is the plain
 * schedule. */
typedef struct {
    int32_t num_layers;         /* N in KV_M(C) = {(K^(1),V^(1)) .. (K^(N),V^(N))} (Section 2.1) */
    int32_t num_kv_heads;       /* KV heads per layer */
    int32_t head_dim;           /* channels per head: 64, 128 or 256 */
    double  rope_base;          /* RoPE base of K; <= 0 means K carries no rotary encoding */
    int32_t rope_type;          /* kvx_rope_type */
    double  rope_factor;        /* LINEAR, LLAMA3: scale factor, > 0 */
    double  rope_low_freq_factor;       /* LLAMA3: > 0 */
    double  rope_high_freq_factor;      /* LLAMA3: > rope_low_freq_factor */
    int32_t rope_original_max_position; /* LLAMA3: context length of the unscaled model, > 0 */
    int32_t rotary_dim;         /* partial rotary heads: only the first rotary_dim channels of K
                                   rotate, as pairs (i, i + rotary_dim/2) with frequencies
                                   base^(-2i/rotary_dim) under the schedule; the other channels
                                   carry no position.  0 = head_dim (the whole head rotates);
                                   else a multiple of 16 in [16, head_dim]. */
} kvx_model_geom;

/* Which source KV heads feed one target KV head.  Section 5 lists the granularities a
 * translator may act on: individual KV heads, individual layers, groups of layers, and
 * low-dimensional latent adapters (kvx_translator_create_low_rank). */
typedef enum {
    KVX_FORM_GROUPED = 0,       /* per KV head: target head h reads its GQA group of source heads
                                   (h*r .. h*r+r-1 with r = src heads / dst heads), or source head
                                   h/e when the target has e times more heads */
    KVX_FORM_DENSE = 1          /* per layer: every target head reads all src.num_kv_heads heads */
} kvx_form;

/* Translator description (the theta of T_theta, Section 5, plus the layer alignment).  A
 * zero-initialised tail (form 0, layers_per_target 0) is the per-KV-head form over one source
 * layer per target layer. */
typedef struct {
    kvx_model_geom src;         /* source model A */
    kvx_model_geom dst;         /* target model B */
    const int32_t* layer_map;   /* host int32[dst.num_layers][k] (k = layers_per_target): the source
                                   layers feeding each target layer, each in [0, src.num_layers);
                                   NULL = nearest relative depth (kvx_layer_map_nearest), k = 1 only */
    int32_t dtype;              /* kvx_dtype of caches and weights */
    int32_t max_position;       /* RoPE positions must lie in [0, max_position); 0 = 1<<24,
                                   at most 1<<30.  Positions outside are clamped and flagged. */
    int32_t path;               /* kvx_path */
    int32_t form;               /* kvx_form */
    int32_t layers_per_target;  /* k: source layers whose heads are concatenated into one target
                                   layer's input (a group of layers); 0 or 1 = one; at most 4,
                                   and dst.num_layers * k <= 256 */
} kvx_translator_desc;

typedef struct kvx_translator kvx_translator;

/* Build a translator.
 *   w_k, w_v: translator matrices, row-major [dst.num_layers][dst.num_kv_heads][in][out] of
 *     desc->dtype, with out = dst.head_dim and in = k * n * src.head_dim: the input row of
 *     target head h concatenates, for each of its k source layers in layer_map order, the n
 *     source heads that feed it in ascending order.  n is r = src.num_kv_heads/dst.num_kv_heads
 *     (heads h*r .. h*r+r-1) in the grouped form when src has at least as many KV heads as dst,
 *     1 (head h / (dst.num_kv_heads/src.num_kv_heads)) in the grouped form otherwise, and
 *     src.num_kv_heads in the dense form.
 *   weights_on_device: 0 = host pointers, 1 = device pointers.
 * The library copies the weights into its own device memory (re-laid out for its kernels) and
 * builds its RoPE tables; the caller may free its copies on return.  Synchronous on the
 * current device.  Returns KVX_ERR_UNSUPPORTED unless one head count divides the other,
 * both head dims are in {64, 128, 256} and in <= 1024, and KVX_ERR_INVALID_ARG for an unknown
 * form or rope_type, out-of-range schedule parameters, or layers_per_target > 1 without a
 * layer_map.  On success *out owns device memory until kvx_destroy. */
KVX_API kvx_status kvx_translator_create(const kvx_translator_desc* desc, const void* w_k, const void* w_v,
                                         int32_t weights_on_device, kvx_translator** out);

/* Build a translator whose matrices are low-dimensional latent adapters (Section 5):
 * W[j,h] = A[j,h] . B[j,h] with A [in][rank] and B [rank][out], applied to the span mean as the
 * two maps x -> x.A -> (x.A).B.
 *   a_k, b_k, a_v, b_v: row-major [dst.num_layers][dst.num_kv_heads][in][rank] (a_*) and
 *     [dst.num_layers][dst.num_kv_heads][rank][out] (b_*) of desc->dtype; host or device per
 *     weights_on_device.  1 <= rank <= 1024.
 * The library multiplies the factors once, on the device (fp32 accumulation over rank, then
 * rounded to desc->dtype), and from then on holds only W: the translation reads the source and
 * writes the target cache at the same HBM cost whatever the rank, so the product costs the
 * kernels nothing, while two chained contractions would add a round trip through on-chip
 * memory.  Everything else is as for kvx_translator_create. */
KVX_API kvx_status kvx_translator_create_low_rank(const kvx_translator_desc* desc, int32_t rank, const void* a_k,
                                                  const void* b_k, const void* a_v, const void* b_v,
                                                  int32_t weights_on_device, kvx_translator** out);

/* Source KV cache KV_A(C) (Section 2.1), one K and one V tensor per source layer, each
 * [batch][src.num_kv_heads][max_seq][src.head_dim] addressed by the strides below with the
 * head_dim channels contiguous.  K holds the source model's post-RoPE keys. */
typedef struct {
    int32_t batch;
    int32_t max_seq;            /* padded tokens per sequence in the source tensors */
    const void* const* k;       /* host array [src.num_layers] of device pointers */
    const void* const* v;       /* host array [src.num_layers] of device pointers */
    int64_t stride_b, stride_h, stride_s;   /* elements; multiples of 8 for bf16, 4 for fp32 */
    const int32_t* seq_len;     /* device int32[batch]: source tokens of each sequence (<= max_seq) */
    const int32_t* pos;         /* device int32[batch*max_seq]: RoPE position of each source token,
                                   or NULL for 0..seq_len-1 */
} kvx_src_kv;

/* Target tokens and their alignment to source tokens.  Target tokens of all sequences are
 * packed: sequence b owns packed indices [seq_off[b], seq_off[b+1]). */
typedef struct {
    int32_t total_tokens;       /* T_total = seq_off[batch] (host copy, sizes the launch) */
    const int32_t* seq_off;     /* device int32[batch+1], seq_off[0] = 0, non-decreasing */
    const int32_t* span_lo;     /* device int32[T_total]: first source token (index within its
                                   sequence) of each target token's span; NULL with span_hi
                                   NULL = identity alignment (span of t is [t, t+1)) */
    const int32_t* span_hi;     /* device int32[T_total]: one past the span's last source token.
                                   With identity alignment a target token at or past its
                                   sequence's source length is flagged (KVX_DEV_SPAN_CLAMPED)
                                   and its output row is unspecified. */
    const int32_t* pos;         /* device int32[T_total]: RoPE position of each target token, or
                                   NULL for its index within its sequence */
} kvx_tgt_tokens;

/* Target KV cache written by kvx_translate: one K and one V tensor per target layer.
 * Contiguous (paged = 0): element (b, h, t, c) at b*stride_b + h*stride_h + t*stride_t + c,
 *   t < max_seq.
 * Paged (paged = 1): pool [num_pages][page_size][dst.num_kv_heads][dst.head_dim]; token t of
 *   sequence b lives in page page_table[b*max_pages_per_seq + t/page_size], slot t%page_size.
 * Rows of padding tokens and of unlisted pages are not touched. */
typedef struct {
    void* const* k;             /* host array [dst.num_layers] of device pointers */
    void* const* v;             /* host array [dst.num_layers] of device pointers */
    int32_t paged;
    int32_t max_seq;                        /* contiguous: token capacity per sequence */
    int64_t stride_b, stride_h, stride_t;   /* contiguous: elements; multiples of 8 (bf16) / 4 (fp32) */
    const int32_t* page_table;              /* paged: device int32[batch*max_pages_per_seq] */
    int32_t max_pages_per_seq;
    int32_t page_size;                      /* paged: tokens per page (16 in the evaluated setups) */
    int32_t num_pages;                      /* paged: pages in the pool */
} kvx_dst_kv;

/* Translate KV_A(C) into the target cache: KV^_B(C) = T_theta(KV_A(C)) (Sections 4 and 5).
 * Asynchronous on stream; allocates nothing; never synchronises.  The source, alignment and
 * position buffers must stay valid and unchanged until the work on stream completes.  Output
 * rows of distinct target tokens are written exactly once.
 * Calls on one translator must be ordered: issue them on one stream, or serialise them on the
 * host and order them on the device (events).  The translator owns per-call state that two
 * overlapping calls would share: the span kernel's plan buffer on the device, the cache of
 * source tensor descriptors and the launch count on the host.  Distinct translators may run
 * concurrently on different streams and host threads. */
KVX_API kvx_status kvx_translate(kvx_translator* tr, const kvx_src_kv* src, const kvx_tgt_tokens* tgt,
                                 const kvx_dst_kv* dst, void* stream);

/* Writing the translation into the target model's GPU.  In the paper's handoff (Section 6.1,
 * Table 4) the source model's GPU translates, a peer-to-peer copy moves the translated state to
 * the target model's GPU, and the target cache is assembled there.  kvx_translate_to_device
 * runs on the source GPU (the current device, which holds the source caches and the translator)
 * and leaves the translated rows in a target cache on dst_device:
 *   KVX_PEER_STORES  the translation kernels write every target row straight into dst (16-byte
 *                    stores issued by the kernel's threads, over the peer mapping when dst_device
 *                    is another GPU): copy and cache assembly fused into the translation; any
 *                    layout (contiguous or paged).  Needs kvx_enable_peer(dst_device) first
 *                    when dst_device is not the current device.
 *   KVX_PEER_STAGED  translate into `staging` (a contiguous cache on the current device with the
 *                    same layout as dst), then one cudaMemcpyPeerAsync per target tensor copies
 *                    its whole [batch][heads][max_seq][head_dim] extent (padding rows included)
 *                    to dst.  Contiguous targets only (KVX_ERR_UNSUPPORTED for paged ones).
 * dst_device equal to the current device is allowed in both modes (the same kernels and copies
 * on one GPU).  Every dst (and staging) tensor must be memory of dst_device (the current
 * device), else KVX_ERR_INVALID_ARG.  Asynchronous on stream; allocates nothing; the ordering
 * rule of kvx_translate applies. */
typedef enum {
    KVX_PEER_STORES = 0,
    KVX_PEER_STAGED = 1
} kvx_peer_mode;

/* Enables access from the current device to peer_device's memory (cudaDeviceEnablePeerAccess;
 * a one-time set-up per device pair, idempotent, to be called outside stream capture).
 * KVX_ERR_UNSUPPORTED when the devices cannot reach each other.  peer_device equal to the
 * current device is accepted and does nothing. */
KVX_API kvx_status kvx_enable_peer(int32_t peer_device);

KVX_API kvx_status kvx_translate_to_device(kvx_translator* tr, const kvx_src_kv* src, const kvx_tgt_tokens* tgt,
                                           const kvx_dst_kv* dst, int32_t dst_device, int32_t mode,
                                           const kvx_dst_kv* staging, void* stream);

/* Token-span alignment from byte offsets (a target token is aligned to the source tokens whose
 * last byte lies in its byte range; a target token that receives none takes the source token
 * holding its own last byte).  Tokenizer differences are among the model differences the
 * paper's translator must bridge (Sections 1 and 4).
 *   src_end: device int32[total_src], tgt_end: device int32[total_tgt]: byte-end offsets of
 *     each token, strictly increasing within a sequence and relative to the sequence start.
 *   src_seq_off, tgt_seq_off: device int32[batch+1] packed offsets.
 *   span_lo, span_hi: device int32[total_tgt] outputs (indices within each sequence).
 *   dev_status: device uint32 or NULL; KVX_DEV_SPAN_CLAMPED is OR-ed in when a target text
 *     runs past the end of its source text (span clamped to the last source token).
 * Asynchronous on stream; allocates nothing. */
KVX_API kvx_status kvx_build_alignment(int32_t batch, int32_t total_src, int32_t total_tgt,
                                       const int32_t* src_seq_off, const int32_t* src_end,
                                       const int32_t* tgt_seq_off, const int32_t* tgt_end,
                                       int32_t* span_lo, int32_t* span_hi, uint32_t* dev_status,
                                       void* stream);

/* Layer alignment: out[j] = the source layer nearest target layer j in relative depth,
 * round(j*(L_s-1)/(L_t-1)) with halves rounded up; out[0] = 0 when L_t = 1.  Host only. */
KVX_API kvx_status kvx_layer_map_nearest(int32_t src_layers, int32_t dst_layers, int32_t* out);

/* Synchronise stream, then read the translator's device status word into *bits (may be NULL)
 * and, if clear != 0, reset it to zero.  Returns KVX_ERR_DEVICE_STATUS when it was nonzero. */
KVX_API kvx_status kvx_get_device_status(kvx_translator* tr, void* stream, uint32_t* bits, int32_t clear);

/* What kvx_translate will launch for this translator. */
typedef struct {
    int32_t path;               /* KVX_PATH_SIMT or KVX_PATH_TCGEN05 */
    int32_t group_in;           /* in: input width of one translator matrix */
    int32_t n_tile;             /* output columns per tensor-core tile (tcgen05) */
    int32_t smem_bytes;         /* dynamic shared memory per CTA */
    int32_t threads;            /* threads per CTA */
    int32_t num_sms;            /* SMs of the device */
    int64_t weight_bytes;       /* device bytes held for weights */
    int64_t table_bytes;        /* device bytes held for RoPE tables */
} kvx_translator_info;

KVX_API kvx_status kvx_get_info(const kvx_translator* tr, kvx_translator_info* info);

/* Kernel launches the most recent kvx_translate call on this translator made (for
 * launch accounting): 1 for the identity-alignment and CUDA-core kernels; 2 per
 * chunk of up to 65536 target tokens for the span kernel (a span-plan launch and the
 * translation launch).  0 before the first call and after a call with no tokens. */
KVX_API int32_t kvx_launches_per_translate(const kvx_translator* tr);

/* Diagnostics of the kernels' bounded waits (the failure-detection path, tested without a GPU
 * fault): the next kvx_translate on this translator bounds every on-chip wait by wait_us
 * microseconds (1 .. 1e6) instead of about a second and, when that call runs the
 * identity-alignment kernel, the kernel's first CTA issues no source copies from its unit-th
 * work unit on, so the waits for them run out.  That call then records KVX_DEV_WAIT_TIMEOUT in
 * the status word, drains the copies it started, frees its tensor memory and returns with its
 * output incomplete; the context stays usable and later calls translate normally.  Applies to
 * the next call only. */
KVX_API kvx_status kvx_debug_stall_next_translate(kvx_translator* tr, int32_t unit, int32_t wait_us);

/* Diagnostics of the token-span plan of the most recent kvx_translate on this translator, when
 * that call ran the span kernel (its last chunk of up to 65536 target tokens).  The span kernel
 * stages the source rows of each 32-token sub-tile as one window of consecutive rows (at most
 * 48); a token whose span lies outside its sub-tile's window (a window cut at the cap, a span
 * in another sequence, a non-monotone span) is gathered from global memory instead.
 *   counts: host int64[4] = {sub-tiles, tokens staged in their window, tokens gathered from
 *   global memory, sub-tiles with at least one such token}.
 * Synchronises stream.  KVX_ERR_INVALID_ARG when the last call did not run the span kernel. */
KVX_API kvx_status kvx_span_plan_stats(kvx_translator* tr, void* stream, int64_t* counts);

/* ------------------------------------------------------------------------------------------
 * Closed-form fit of a linear translator (Section 5).  The paper gives the learning objective
 * L_KV = D(T_theta(KV_A(C)), KV_B(C)): the distance between the translated cache and the cache
 * the target's own prefill builds for the same context.  With D the squared Euclidean distance
 * summed over target tokens plus a ridge term lambda |W|^2, and the linear T_theta of
 * kvx_translate, every (target layer j, target head h, K|V) is an independent least-squares
 * problem with the closed-form solution
 *     W[j,h] = (X^T X + lambda I)^{-1} X^T Y,
 * where row t of X is the translator's input row for target token t (the span mean of the
 * un-rotated source rows, exactly as kvx_translate forms it, rounded to the cache dtype) and
 * row t of Y is the target model's own cache row of token t with the target RoPE undone (K;
 * the rotation is orthogonal, so the distance is unchanged) or as stored (V).
 * The fitter accumulates X^T X and X^T Y over any number of calibration calls in fp32 sums (on the
 * tensor cores for bf16 caches with in + out <= 512 and in a multiple of 128, X and Y built on
 * chip; on the CUDA cores otherwise), then solves all systems at once (Cholesky factorisation on
 * the device: in fp32 shared memory for in <= 256, where a system whose factor shows a condition
 * number above 1e3 is factored again in double; in double above).  Forms as for
 * kvx_translator_create; latent adapters are not fitted (fit W, then factor it if wanted). */
typedef struct kvx_fitter kvx_fitter;

/* desc: the translator to fit (its dtype is the cache dtype; desc->path is ignored).
 * lambda: ridge weight, >= 0 (0 needs at least `in` well-spread tokens per system).
 * chunk_tokens: target tokens one accumulation pass handles (calls longer than this run in
 *   several passes); 0 = 4096.  The fitter holds (L_t * H_t * 2) * chunk_tokens * (in + out)
 *   cache-dtype elements of row workspace (none on the tensor-core path) plus the fp32 sums.
 * Requires in <= 512.  Synchronous; on success *out owns device memory until kvx_fit_destroy. */
KVX_API kvx_status kvx_fit_create(const kvx_translator_desc* desc, double lambda, int32_t chunk_tokens,
                                  kvx_fitter** out);

/* Add one calibration batch: source caches, the token alignment, and the target model's own
 * caches for the same context (read-only here; same layouts as for kvx_translate, contiguous
 * or paged).  Target rows that fall outside the target cache (a bad page, t >= max_seq) are
 * left out of the sums and flagged in the fitter's status word.  Asynchronous on stream;
 * allocates nothing. */
KVX_API kvx_status kvx_fit_accumulate(kvx_fitter* f, const kvx_src_kv* src, const kvx_tgt_tokens* tgt,
                                      const kvx_dst_kv* target_cache, void* stream);

/* Solve every system from the sums so far and write W_K and W_V as DEVICE arrays
 * [dst.num_layers][dst.num_kv_heads][in][out] of the desc dtype (the layout
 * kvx_translator_create takes).  Synchronises stream.  status_bits (host, may be NULL) receives
 * the fitter's status word: KVX_DEV_* bits from the accumulation passes (rows left out), 0x20
 * when a system was not positive definite (lambda = 0 with too few tokens; its W is zero), in
 * which case the call returns KVX_ERR_DEVICE_STATUS, and 0x40 (informational) when
 * ill-conditioned systems were factored in double.  Calls on one fitter must be ordered
 * (one stream, or synchronised by the caller). */
KVX_API kvx_status kvx_fit_solve(kvx_fitter* f, void* w_k, void* w_v, uint32_t* status_bits, void* stream);

/* Clear the accumulated sums (start a new fit with the same fitter). */
KVX_API kvx_status kvx_fit_reset(kvx_fitter* f, void* stream);

/* Tokens accumulated so far (sum of total_tokens over kvx_fit_accumulate calls). */
KVX_API int64_t kvx_fit_tokens(const kvx_fitter* f);

/* Free the fitter.  Synchronises the device first.  NULL is accepted. */
KVX_API kvx_status kvx_fit_destroy(kvx_fitter* f);

/* Size of the device scratch array kvx_translate_static works in (8 MiB). */
#define KVX_STATIC_SCRATCH_BYTES (8u << 20)

/* Translate without allocating device memory.  The paper has no counterpart; this exists for
 * callers that cannot call cudaMalloc when they translate: a serving process whose device memory
 * belongs to a caching allocator that forbids raw allocations, a runtime whose memory budget is
 * fixed at start-up, or a latency-critical path where cudaMalloc/cudaFree would synchronise the
 * device.  kvx_translator_create allocates; this call does not.
 *
 * It runs the CUDA-core translation kernel (the KVX_PATH_SIMT path of kvx_translate) with its
 * scratch (status word, rotation frequencies and the weights) in one file-scope device array of
 * KVX_STATIC_SCRATCH_BYTES, which every GPU that loads the library holds until the process exits.
 * The arguments mean what they mean for kvx_translator_create and kvx_translate, except:
 *   w_k, w_v: DEVICE pointers, row-major [dst.num_layers][dst.num_kv_heads][in][out] of
 *     desc->dtype; they are copied into the scratch array on every call.  Both together must fit
 *     KVX_STATIC_SCRATCH_BYTES minus 2304 bytes, else KVX_ERR_UNSUPPORTED (nothing is launched).
 *   desc->path is ignored; desc->form must be KVX_FORM_GROUPED and desc->layers_per_target at
 *     most 1, and the translator input width (r * src.head_dim, or src.head_dim when the target
 *     has more KV heads) at most 512 (else KVX_ERR_UNSUPPORTED).  Paged targets are accepted.
 *   status_bits: host pointer or NULL.  If set, the call synchronises stream, writes the device
 *     status word there and returns KVX_ERR_DEVICE_STATUS when it is nonzero; if NULL, the call is
 *     asynchronous on stream like kvx_translate.
 * The first call on a device looks up the array's device address with that device current (a
 * one-time set-up, repeated when a call finds another driver context current than the one of
 * the lookup, e.g. after cudaDeviceReset); make that first call before any stream capture.  Every call shares the one
 * array and clears the status word itself, so calls that overlap on the GPU (different streams,
 * or several host threads) race on the scratch and must be serialised by the caller.
 * Calls no cudaMalloc, cudaFree or other allocating routine.  Errors: kvx_static_last_error(). */
KVX_API kvx_status kvx_translate_static(const kvx_translator_desc* desc, const void* w_k, const void* w_v,
                                        const kvx_src_kv* src, const kvx_tgt_tokens* tgt, const kvx_dst_kv* dst,
                                        uint32_t* status_bits, void* stream);

/* Message of the last failed kvx_translate_static call on this thread ("" if none). */
KVX_API const char* kvx_static_last_error(void);

/* Message of the last failed call on this thread ("" if none). */
KVX_API const char* kvx_last_error(void);

/* Free the translator's device memory.  Synchronises the device first.  NULL is accepted. */
KVX_API kvx_status kvx_destroy(kvx_translator* tr);

#ifdef __cplusplus
}
#endif
#endif /* KVX_H */
