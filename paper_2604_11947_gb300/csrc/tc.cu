// tc.cu -- sm_103a tensor-core kernels of the ResBM boundary bottleneck.
#include "tc.h"

namespace resbm {

bool tc_supported(const resbm_desc &, int) { return false; }
size_t tc_ws_bytes(const resbm_desc &, int) { return 0; }

cudaError_t tc_encode_fwd(const resbm_desc &, const void *, const void *, const void *,
                          const void *, void *, float *, void *, const Ctx &)
{
    return cudaErrorNotSupported;
}
cudaError_t tc_decode_fwd(const resbm_desc &, const void *, const void *, const void *, void *,
                          void *, const Ctx &)
{
    return cudaErrorNotSupported;
}
cudaError_t tc_decode_bwd(const resbm_desc &, const void *, const void *, const void *,
                          const void *, void *, float *, float *, void *, const Ctx &)
{
    return cudaErrorNotSupported;
}
cudaError_t tc_encode_bwd(const resbm_desc &, const void *, const void *, const float *,
                          const void *, const void *, void *, void *, float *, float *, void *,
                          const Ctx &)
{
    return cudaErrorNotSupported;
}

}  // namespace resbm
