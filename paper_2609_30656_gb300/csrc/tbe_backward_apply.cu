// tbe_backward_apply.cu -- the segmented reduce with the optimizer step fused
// in place of the gradient output, for fp32 grad_out (the kernels of
// tbe_reduce.cuh with APPLY).
#include "tbe_reduce.cuh"

namespace cbtbe {

void launch_bwd_reduce_f32_apply(const Problem& P, const Plan& Q, const BwdOut& O, const void* grad_out,
                                 int cls, int vpl, int gc, bool packed, int64_t chunk_bound, int num_sms,
                                 cudaStream_t s) {
    launch_bwd_reduce_t<CB_F32, true>(P, Q, O, grad_out, cls, vpl, gc, packed, chunk_bound, num_sms, s);
}

}  // namespace cbtbe
