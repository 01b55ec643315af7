// tbe_forward_f32.cu -- forward gather-pool instantiations for f32 tables.
#include "tbe_forward.cuh"

namespace cbtbe {

void launch_fwd_gather_f32(const Problem& P, const Plan& Q, void* out, int cls, int vpl, int gc,
                           int64_t chunk_bound, int num_sms, cudaStream_t s) {
    launch_gather_dtype<CB_F32>(P, Q, out, cls, vpl, gc, chunk_bound, num_sms, s);
}

}  // namespace cbtbe
