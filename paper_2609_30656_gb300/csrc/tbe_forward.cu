// tbe_forward.cu -- forward fix-up (bags split across chunks) and the launch
// switch over storage types; the gather-pool kernel is in tbe_forward.cuh.
#include "tbe_internal.cuh"
#include "tbe_launch.h"

namespace cbtbe {

// A heavy bag split over chunks: its tail piece (chunk where it starts) plus the
// head pieces of the following chunks, added in fp64, then scaled. Each warp
// scans 32 chunks at a time for tails (rare once boundaries snap to bag ends).
__global__ void __launch_bounds__(kWarpThreads) fwd_fixup_kernel(const __grid_constant__ Problem P,
                                                                 const __grid_constant__ Plan Q,
                                                                 void* out) {
    const int lane = threadIdx.x & 31;
    const int64_t total = min64(Q.class_chunk_base[Q.num_classes], Q.max_chunks);
    for (int64_t base = warp_id_global() * 32; base < total; base += warps_in_grid() * 32) {
        const int64_t mine = base + lane < total ? Q.tail_owner[base + lane] : -1;
        for (uint32_t mask = __ballot_sync(kFull, mine >= 0); mask; mask &= mask - 1) {
            const int b = __ffs(mask) - 1;
            const int64_t j = base + b;
            const int64_t bag = __shfl_sync(kFull, mine, b);
            const int t = Q.chunks[j].table;
            const TableDev& td = P.tables[t];
            const int64_t s = load_index(P.offsets, bag, P.is32);
            const int64_t e = load_index(P.offsets, bag + 1, P.is32);
            const int64_t m = pieces_after(Q, j, e, total);
            const double L = (P.mean && e > s) ? static_cast<double>(e - s) : 0.0;
            const int64_t col0 = (bag - static_cast<int64_t>(t) * P.B) * P.sum_d + td.doff;
            combine_pieces(Q, j, m, td.dim, P.dmax, lane, [&](int x0, double (&acc)[4]) {
                if (L > 0.0)
                    for (int x = 0; x < 4; ++x) acc[x] /= L;
                store_out4(out, col0 + x0, static_cast<float>(acc[0]), static_cast<float>(acc[1]),
                           static_cast<float>(acc[2]), static_cast<float>(acc[3]), P.out_dtype);
            });
        }
    }
}

void launch_fwd_gather_f32(const Problem&, const Plan&, void*, int, int, int, int64_t, int,
                           cudaStream_t);
void launch_fwd_gather_f16(const Problem&, const Plan&, void*, int, int, int, int64_t, int,
                           cudaStream_t);
void launch_fwd_gather_bf16(const Problem&, const Plan&, void*, int, int, int, int64_t, int,
                            cudaStream_t);

void launch_fwd_gather(const Problem& P, const Plan& Q, void* out, int cls, int dtype, int vpl,
                       int gc, int64_t chunk_bound, int num_sms, cudaStream_t s) {
    if (dtype == CB_F32) launch_fwd_gather_f32(P, Q, out, cls, vpl, gc, chunk_bound, num_sms, s);
    else if (dtype == CB_F16) launch_fwd_gather_f16(P, Q, out, cls, vpl, gc, chunk_bound, num_sms, s);
    else launch_fwd_gather_bf16(P, Q, out, cls, vpl, gc, chunk_bound, num_sms, s);
}

void launch_fwd_fixup(const Problem& P, const Plan& Q, void* out, int64_t chunk_bound,
                      int num_sms, cudaStream_t s) {
    const int64_t need = (chunk_bound + kWarpThreads - 1) / kWarpThreads;  // 32 chunks per warp
    const int grid = static_cast<int>(max64(1, min64(need, static_cast<int64_t>(num_sms) * 8)));
    fwd_fixup_kernel<<<grid, kWarpThreads, 0, s>>>(P, Q, out);
}

}  // namespace cbtbe
