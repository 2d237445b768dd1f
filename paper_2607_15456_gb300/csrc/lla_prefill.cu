// lla_prefill.cu -- causal pass-2 prefill attention over latents.
#include "lla_internal.h"

namespace lla {

lla_status launch_prefill(const PrefillArgs &, cudaStream_t) { return LLA_ERR_UNSUPPORTED; }

}  // namespace lla
