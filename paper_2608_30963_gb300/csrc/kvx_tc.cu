// kvx_tc.cu -- tensor-core (tcgen05/TMEM) translation kernel.  Placeholder: not yet built.
#include "kvx_common.cuh"
#include "kvx_kernels.h"

namespace kvx {
TcConfig tc_config(int, int, int) { return TcConfig{0, 0, 0, 0, 0}; }
size_t tc_weight_image_bytes(int, int, int, int) { return 0; }
cudaError_t launch_tc_weight_relayout(const void*, const void*, void*, int, int, int, int, int, cudaStream_t)
{
    return cudaErrorNotSupported;
}
cudaError_t launch_translate_tc(const TranslateParams&, const TcConfig&, int, cudaStream_t)
{
    return cudaErrorNotSupported;
}
}  // namespace kvx
