// prefill.cu -- placeholder until the tcgen05 prefill kernel lands.
#include "pkv_internal.h"
namespace pkv {
cudaError_t launch_prefill(const PrefillArgs &, cudaStream_t, Tracer *) { return cudaErrorNotSupported; }
}  // namespace pkv
