// tbe_forward_bf16.cu -- forward gather-pool instantiations for bf16 tables.
#include "tbe_forward.cuh"

namespace cbtbe {

void launch_fwd_gather_bf16(const Problem& P, const Plan& Q, void* out, int cls, int vpl, int gc,
                           int64_t chunk_bound, int num_sms, cudaStream_t s) {
    launch_gather_dtype<CB_BF16>(P, Q, out, cls, vpl, gc, chunk_bound, num_sms, s);
}

}  // namespace cbtbe
