// kvx_kernels.h -- launchers of the kvx CUDA kernels (library-internal).
#pragma once
#include <cuda_runtime.h>
#include <stddef.h>

namespace kvx {
struct TranslateParams;

size_t simt_smem_bytes(int in_dim, int dt);
cudaError_t launch_translate_simt(const TranslateParams& P, int dtype, cudaStream_t stream);
// W = A . B for n (layer, head, K|V) matrices (latent adapters, at translator creation)
cudaError_t launch_fold_low_rank(const void* a, const void* b, void* w, int n, int in_dim, int rank, int out,
                                 int dtype, cudaStream_t stream);

cudaError_t launch_build_alignment(int batch, int total_tgt, const int* src_seq_off, const int* src_end,
                                   const int* tgt_seq_off, const int* tgt_end, int* span_lo, int* span_hi,
                                   unsigned* status, cudaStream_t stream);


// tensor-core path
struct TcConfig {
    int n_tile;        // output columns per MMA tile
    int n_split;       // d_t / n_tile
    int smem_bytes;
    int threads;
    int ok;            // geometry supported
};
// share: target heads that read the same input rows (share_heads); it decides how many heads
// one unit of the span kernel covers and so the weight images' output split n_tile.
TcConfig tc_config(int in_dim, int dt, int ds, int share);
size_t tc_weight_image_bytes(int in_dim, int dt, int Lt, int Ht);
// rhalf_t: rotating pairs of the target head (rotary_dim/2; d_t/2 unless partial rotary)
cudaError_t launch_tc_weight_relayout(const void* w_k, const void* w_v, void* image, int Lt, int Ht, int in_dim,
                                      int dt, int n_tile, int rhalf_t, cudaStream_t stream);
size_t tc_plan_bytes(int tokens);
// Where the plan of the last chunk of a span-kernel call lives in the plan buffer: its
// sub-tile headers start at int4 0, its per-token entries (32 per sub-tile) at int4
// *ent_off; *nsub sub-tiles.  T_total: target tokens of the call.
void tc_plan_layout(int T_total, int plan_tokens, int* nsub, int* ent_off);
// One span-plan launch and one translation launch per chunk of at most plan_tokens
// target tokens; *launches receives the number of launches made.
cudaError_t launch_translate_tc(const TranslateParams& P, const TcConfig& cfg, int num_sms, void* plan,
                                int plan_tokens, cudaStream_t stream, int* launches);

// identity-alignment tensor-core path (tensor-TMA fed)
bool aligned_supported(int in_dim, int dt, int ds, int share, int Lt, int batch, int kl);
size_t aligned_map_bytes();
bool encode_source_map(void* map_out, const void* base, int ds, int S_max, int Hs, int batch, long long ss,
                       long long sh, long long sb);
cudaError_t launch_translate_tc_aligned(const TranslateParams& P, const void* const* maps,
                                        const unsigned long long* host_turns, int num_sms, cudaStream_t stream);
}  // namespace kvx
