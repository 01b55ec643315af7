// tbe_reduce_bf16.cu -- the segmented reduce (and its fused optimizer step) for
// bf16 grad_out, the mixed-precision backward: rows gathered in bf16, summed
// in fp32 (the kernels of tbe_reduce.cuh).
#include "tbe_reduce.cuh"

namespace cbtbe {

void launch_bwd_reduce_bf16(const Problem& P, const Plan& Q, const BwdOut& O, const void* grad_out, int cls,
                          int vpl, int gc, bool packed, bool apply, int64_t chunk_bound, int num_sms,
                          cudaStream_t s) {
    if (apply)
        launch_bwd_reduce_t<CB_BF16, true>(P, Q, O, grad_out, cls, vpl, gc, packed, chunk_bound, num_sms, s);
    else
        launch_bwd_reduce_t<CB_BF16, false>(P, Q, O, grad_out, cls, vpl, gc, packed, chunk_bound, num_sms, s);
}

}  // namespace cbtbe
