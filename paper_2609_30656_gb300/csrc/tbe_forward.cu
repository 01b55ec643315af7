// tbe_forward.cu -- forward fix-up (bags split across chunks) and the launch
// switch over storage types; the gather-pool kernel is in tbe_forward.cuh.
#include "tbe_internal.cuh"
#include "tbe_launch.h"

namespace cbtbe {

// A bag split over chunks: its tail piece (chunk where it starts) plus the head
// pieces of the following chunks, added in fp64, then scaled. One warp per chunk.
__global__ void __launch_bounds__(kWarpThreads) fwd_fixup_kernel(const __grid_constant__ Problem P,
                                                                 const __grid_constant__ Plan Q,
                                                                 float* out) {
    const int lane = threadIdx.x & 31;
    const int64_t total = min64(Q.class_chunk_base[Q.num_classes], Q.max_chunks);
    const int64_t j = warp_id_global();
    if (j >= total) return;
    const int64_t bag = Q.tail_owner[j];
    if (bag < 0) return;
    const int t = Q.chunks[j].table;
    const TableDev& td = P.tables[t];
    const int64_t s = load_index(P.offsets, bag, P.is32);
    const int64_t e = load_index(P.offsets, bag + 1, P.is32);
    const int64_t m = pieces_after(Q, j, e, total);
    const double L = (P.mean && e > s) ? static_cast<double>(e - s) : 0.0;
    float* dst = out + (bag - static_cast<int64_t>(t) * P.B) * P.sum_d + td.doff;
    combine_pieces(Q, j, m, td.dim, P.dmax, lane, [&](int x0, double (&acc)[4]) {
        if (L > 0.0)
            for (int x = 0; x < 4; ++x) acc[x] /= L;
        *reinterpret_cast<float4*>(dst + x0) =
            make_float4(static_cast<float>(acc[0]), static_cast<float>(acc[1]),
                        static_cast<float>(acc[2]), static_cast<float>(acc[3]));
    });
}

void launch_fwd_gather_f32(const Problem&, const Plan&, float*, int, int, int, int64_t, int,
                           cudaStream_t);
void launch_fwd_gather_f16(const Problem&, const Plan&, float*, int, int, int, int64_t, int,
                           cudaStream_t);
void launch_fwd_gather_bf16(const Problem&, const Plan&, float*, int, int, int, int64_t, int,
                            cudaStream_t);

void launch_fwd_gather(const Problem& P, const Plan& Q, float* out, int cls, int dtype, int vpl,
                       int gc, int64_t chunk_bound, int num_sms, cudaStream_t s) {
    if (dtype == CB_F32) launch_fwd_gather_f32(P, Q, out, cls, vpl, gc, chunk_bound, num_sms, s);
    else if (dtype == CB_F16) launch_fwd_gather_f16(P, Q, out, cls, vpl, gc, chunk_bound, num_sms, s);
    else launch_fwd_gather_bf16(P, Q, out, cls, vpl, gc, chunk_bound, num_sms, s);
}

void launch_fwd_fixup(const Problem& P, const Plan& Q, float* out, int64_t chunk_bound,
                      int num_sms, cudaStream_t s) {
    (void)num_sms;  // one warp per chunk
    const int64_t need = (chunk_bound + (kWarpThreads / 32) - 1) / (kWarpThreads / 32);
    fwd_fixup_kernel<<<static_cast<unsigned>(max64(need, 1)), kWarpThreads, 0, s>>>(P, Q, out);
}

}  // namespace cbtbe
