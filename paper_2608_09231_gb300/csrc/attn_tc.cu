// Tensor-core (tcgen05) flash attention: placeholder until the kernel lands.
#include "kernels.h"

namespace bag {

cudaError_t attention_tc_init() { return cudaSuccess; }
int attention_tc_supported(const AttnArgs&) { return 0; }
cudaError_t attention_tc(const AttnArgs&, int*, cudaStream_t) { return cudaErrorNotSupported; }

}  // namespace bag
