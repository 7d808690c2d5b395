// Causal prefill attention (tcgen05 / TMEM / TMA): not built yet.
#include "kernels.h"

namespace tk {
cudaError_t launch_prefill(const PrefillParams&, cudaStream_t, int* unsupported) {
  *unsupported = 1;
  return cudaSuccess;
}
}  // namespace tk
