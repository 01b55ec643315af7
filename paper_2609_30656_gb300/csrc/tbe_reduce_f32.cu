// tbe_reduce_f32.cu -- the segmented reduce that writes gradients, for fp32
// grad_out (the kernels of tbe_reduce.cuh without the optimizer step).
#include "tbe_reduce.cuh"

namespace cbtbe {

void launch_bwd_reduce_f32(const Problem& P, const Plan& Q, const BwdOut& O, const void* grad_out, int cls,
                           int vpl, int gc, bool packed, int64_t chunk_bound, int num_sms, cudaStream_t s) {
    launch_bwd_reduce_t<CB_F32, false>(P, Q, O, grad_out, cls, vpl, gc, packed, chunk_bound, num_sms, s);
}

}  // namespace cbtbe
