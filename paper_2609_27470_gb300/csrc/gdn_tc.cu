// Tensor-core (tcgen05 / TMEM / TMA) gated-delta-rule chunk update for d = 128, bfloat16.
#include "internal.cuh"

namespace deltas {

bool gdn_tc_supported(const GdnArgs& a) {
    (void)a;
    return false;
}

cudaError_t launch_gdn_update_tc(const GdnArgs& a, cudaStream_t s) {
    (void)a; (void)s;
    return cudaErrorNotSupported;
}

}  // namespace deltas
