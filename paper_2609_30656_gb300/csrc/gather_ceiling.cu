// gather_ceiling.cu -- cb_gather_ceiling: the random-row gather rate of this GPU
// for a set of rows that fits in L2, measured with the load shape of the
// library's walkers and none of their segment bookkeeping.
//
// On skewed (Zipf) indices most rows the forward gather and the backward
// reduce read are served from L2, not HBM, so the rate at which a warp can
// gather random 16-byte-per-lane rows out of L2 bounds those kernels, and their
// time is judged against it as well as against the HBM copy bandwidth. Each
// warp takes 32 items at a time (one coalesced 4-byte index load per lane, as
// the reduce reads its payloads), gathers their rows G per warp step with
// kRows steps of loads in flight, and sums everything it loaded; the sum of
// each 32-item batch is written so the loads cannot be dropped and the result
// can be checked.
#include <cstdint>

#include "cb_tbe.h"
#include "tbe_internal.cuh"
#include "tbe_reduce.cuh"

namespace cbtbe {
namespace {

constexpr int kRows = 8;  // row steps in flight per lane (the fp32 reduce's setting)

template <int G>
__global__ void __launch_bounds__(kWarpThreads) gather_ceiling_kernel(const uint4* __restrict__ rows,
                                                                      uint32_t stride, int64_t num_rows,
                                                                      const uint32_t* __restrict__ idx,
                                                                      int64_t n, float* __restrict__ out) {
    constexpr int V = 32 / G;            // lanes per row
    constexpr int kSteps = 32 / G;       // row steps per batch of 32 items
    constexpr int UG = kRows < kSteps ? kRows : kSteps;
    const int lane = threadIdx.x & 31;
    const int g = lane / V, v = lane - g * V;
    const int64_t batches = (n + 31) / 32;
    for (int64_t b = warp_id_global(); b < batches; b += warps_in_grid()) {
        const int64_t q = b * 32 + lane;
        uint32_t my = q < n ? __ldg(idx + q) : 0u;
        if (my >= num_rows) my = 0;  // kept inside the row set whatever the indices hold
        const bool live = q < n;
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int s0 = 0; s0 < kSteps; s0 += UG) {
            uint4 x[UG];
            bool ok[UG];
#pragma unroll
            for (int u = 0; u < UG; ++u) {
                const int src = (s0 + u) * G + g;
                const uint32_t r = __shfl_sync(kFull, my, src);
                ok[u] = __shfl_sync(kFull, live, src);
                x[u] = __ldg(rows + static_cast<uint64_t>(r) * stride + v);
            }
#pragma unroll
            for (int u = 0; u < UG; ++u) {
                if (!ok[u]) continue;
                acc[0] += __uint_as_float(x[u].x);
                acc[1] += __uint_as_float(x[u].y);
                acc[2] += __uint_as_float(x[u].z);
                acc[3] += __uint_as_float(x[u].w);
            }
        }
        float t = (acc[0] + acc[1]) + (acc[2] + acc[3]);
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) t += __shfl_xor_sync(kFull, t, off);
        if (lane == 0) out[b] = t;
    }
}

template <int G>
cb_status launch(const void* rows, int64_t num_rows, int32_t row_bytes, const uint32_t* idx, int64_t n,
                 float* out, cudaStream_t s) {
    int dev = 0, sms = 1;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
        cudaGetLastError();
        return CB_ERR_CUDA;
    }
    const int cap = occupancy_grid(gather_ceiling_kernel<G>, kWarpThreads, sms);
    const int64_t need = ((n + 31) / 32 + (kWarpThreads / 32) - 1) / (kWarpThreads / 32);
    const int grid = static_cast<int>(need < cap ? (need > 0 ? need : 1) : cap);
    gather_ceiling_kernel<G><<<grid, kWarpThreads, 0, s>>>(static_cast<const uint4*>(rows),
                                                            static_cast<uint32_t>(row_bytes / 16), num_rows,
                                                            idx, n, out);
    return cudaGetLastError() == cudaSuccess ? CB_OK : CB_ERR_CUDA;
}

}  // namespace
}  // namespace cbtbe

extern "C" cb_status cb_gather_ceiling(const void* rows, int64_t num_rows, int32_t row_bytes,
                                       const uint32_t* indices, int64_t num_indices, float* out,
                                       cudaStream_t stream) {
    using namespace cbtbe;
    if (!rows || num_rows <= 0 || num_rows > (int64_t(1) << 32) || num_indices < 0 ||
        (num_indices > 0 && (!indices || !out)) || (reinterpret_cast<uintptr_t>(rows) & 15u))
        return CB_ERR_INVALID_ARG;
    if (num_indices == 0) return CB_OK;
    switch (row_bytes) {
        case 512: return launch<1>(rows, num_rows, row_bytes, indices, num_indices, out, stream);
        case 256: return launch<2>(rows, num_rows, row_bytes, indices, num_indices, out, stream);
        case 128: return launch<4>(rows, num_rows, row_bytes, indices, num_indices, out, stream);
        case 64: return launch<8>(rows, num_rows, row_bytes, indices, num_indices, out, stream);
        default: return CB_ERR_INVALID_ARG;
    }
}
