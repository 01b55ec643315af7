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

#include <cuda.h>
#include <cudaTypedefs.h>

#include "cb_tbe.h"
#include "tbe_internal.cuh"
#include "tbe_reduce.cuh"

namespace cbtbe {
namespace {

// Row steps in flight per lane, and resident blocks per SM the kernel is
// compiled for: the rate out of L2 grows with the warps resident per SM more
// than with the loads each warp has in flight (measured: 4 steps at 8 blocks of
// 256 threads reach ~21 TB/s for 256-byte rows, fp32 or widened fp16, where 8
// steps at 4-5 blocks, the register budget of the walkers, reach 15.8-20 TB/s).
constexpr int kRows = 4;
constexpr int kProbeBlocks = 8;  // 32 registers per thread

// x's values added into acc: fp32 adds, or fp16 values widened into the fp32
// sums by the mixed-precision add (as the forward gather adds them).
template <int DT>
__device__ __forceinline__ void add_row(float (&acc)[DT == CB_F32 ? 4 : 8], const uint4& x) {
    const uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        if constexpr (DT == CB_F32) {
            acc[i] += __uint_as_float(w[i]);
        } else {
            asm("{ .reg .b16 lo, hi;\n\t mov.b32 {lo, hi}, %2;\n\t"
                " add.rn.f32.f16 %0, lo, %0;\n\t add.rn.f32.f16 %1, hi, %1; }"
                : "+f"(acc[2 * i]), "+f"(acc[2 * i + 1]) : "r"(w[i]));
        }
    }
}

// The sum of every value of the rows of one batch of 32 items, per lane
// (lane-summed by the caller). TAIL: the last, partial batch, whose missing
// items add nothing.
template <int G, int DT, bool TAIL>
__device__ __forceinline__ float batch_sum(const uint4* __restrict__ rows, uint32_t my, bool live, int lane) {
    constexpr int V = 32 / G;            // lanes per row
    constexpr int kSteps = 32 / G;       // row steps per batch of 32 items
    constexpr int UG = kRows < kSteps ? kRows : kSteps;
    constexpr int E = DT == CB_F32 ? 4 : 8;
    const int g = lane / V, v = lane - g * V;
    float acc[E];
#pragma unroll
    for (int e = 0; e < E; ++e) acc[e] = 0.f;
#pragma unroll
    for (int s0 = 0; s0 < kSteps; s0 += UG) {
        uint4 x[UG];
        bool ok[UG];
#pragma unroll
        for (int u = 0; u < UG; ++u) {
            const int src = (s0 + u) * G + g;
            const uint32_t r = __shfl_sync(kFull, my, src);
            ok[u] = TAIL ? __shfl_sync(kFull, live, src) : true;
            x[u] = __ldg(rows + static_cast<uint64_t>(r) * V + v);  // a row is V vectors
        }
#pragma unroll
        for (int u = 0; u < UG; ++u)
            if (!TAIL || ok[u]) add_row<DT>(acc, x[u]);
    }
    float t = 0.f;
#pragma unroll
    for (int e = 0; e < E; ++e) t += acc[e];
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) t += __shfl_xor_sync(kFull, t, off);
    return t;
}

// DT: CB_F32 rows summed with fp32 adds (the reduce's grad_out slices), or
// CB_F16 rows widened into fp32 sums by the mixed-precision add, the
// forward's arithmetic on half-precision tables (8 adds per 16 bytes).
// Full batches only; the partial last batch goes to gather_tail_kernel.
template <int G, int DT>
__global__ void __launch_bounds__(kWarpThreads, kProbeBlocks) gather_ceiling_kernel(const uint4* __restrict__ rows,
                                                                      int64_t num_rows,
                                                                      const uint32_t* __restrict__ idx,
                                                                      int64_t batches, float* __restrict__ out) {
    const int lane = threadIdx.x & 31;
    const int64_t warps = static_cast<int64_t>(gridDim.x) * (kWarpThreads / 32);
    for (int64_t b = (static_cast<int64_t>(blockIdx.x) * kWarpThreads + threadIdx.x) / 32; b < batches; b += warps) {
        uint32_t my = __ldg(idx + b * 32 + lane);
        if (my >= num_rows) my = 0;  // kept inside the row set whatever the indices hold
        const float t = batch_sum<G, DT, false>(rows, my, true, lane);
        if (lane == 0) out[b] = t;
    }
}

template <int G, int DT>
__global__ void __launch_bounds__(32) gather_tail_kernel(const uint4* __restrict__ rows, int64_t num_rows,
                                                         const uint32_t* __restrict__ idx, int64_t b, int64_t n,
                                                         float* __restrict__ out) {
    const int lane = threadIdx.x;
    const int64_t q = b * 32 + lane;
    uint32_t my = q < n ? __ldg(idx + q) : 0u;
    if (my >= num_rows) my = 0;
    const float t = batch_sum<G, DT, true>(rows, my, q < n, lane);
    if (lane == 0) out[b] = t;
}

template <int G, int DT>
cb_status launch(const void* rows, int64_t num_rows, int32_t row_bytes, const uint32_t* idx, int64_t n,
                 float* out, cudaStream_t s) {
    int dev = 0, sms = 1;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
        cudaGetLastError();
        return CB_ERR_CUDA;
    }
    // rows of row_bytes = (32 / G) * 16: full batches, then the partial last one
    const uint4* r = static_cast<const uint4*>(rows);
    const int64_t full = n / 32;
    if (full > 0) {
        const int cap = occupancy_grid(gather_ceiling_kernel<G, DT>, kWarpThreads, sms);
        const int64_t need = (full + (kWarpThreads / 32) - 1) / (kWarpThreads / 32);
        const int grid = static_cast<int>(need < cap ? need : cap);
        gather_ceiling_kernel<G, DT><<<grid, kWarpThreads, 0, s>>>(r, num_rows, idx, full, out);
    }
    if (n % 32) gather_tail_kernel<G, DT><<<1, 32, 0, s>>>(r, num_rows, idx, full, n, out);
    return cudaGetLastError() == cudaSuccess ? CB_OK : CB_ERR_CUDA;
}

}  // namespace
}  // namespace cbtbe

namespace cbtbe {
namespace {

template <int DT>
cb_status gather_ceiling(const void* rows, int64_t num_rows, int32_t row_bytes, const uint32_t* indices,
                         int64_t num_indices, float* out, cudaStream_t stream) {
    if (!rows || num_rows <= 0 || num_rows > (int64_t(1) << 32) || num_indices < 0 ||
        (num_indices > 0 && (!indices || !out)) || (reinterpret_cast<uintptr_t>(rows) & 15u))
        return CB_ERR_INVALID_ARG;
    if (num_indices == 0) return CB_OK;
    switch (row_bytes) {
        case 512: return launch<1, DT>(rows, num_rows, row_bytes, indices, num_indices, out, stream);
        case 256: return launch<2, DT>(rows, num_rows, row_bytes, indices, num_indices, out, stream);
        case 128: return launch<4, DT>(rows, num_rows, row_bytes, indices, num_indices, out, stream);
        case 64: return launch<8, DT>(rows, num_rows, row_bytes, indices, num_indices, out, stream);
        default: return CB_ERR_INVALID_ARG;
    }
}

}  // namespace
}  // namespace cbtbe

extern "C" cb_status cb_gather_ceiling(const void* rows, int64_t num_rows, int32_t row_bytes,
                                       const uint32_t* indices, int64_t num_indices, float* out,
                                       cudaStream_t stream) {
    return cbtbe::gather_ceiling<CB_F32>(rows, num_rows, row_bytes, indices, num_indices, out, stream);
}

extern "C" cb_status cb_gather_ceiling_f16(const void* rows, int64_t num_rows, int32_t row_bytes,
                                           const uint32_t* indices, int64_t num_indices, float* out,
                                           cudaStream_t stream) {
    return cbtbe::gather_ceiling<CB_F16>(rows, num_rows, row_bytes, indices, num_indices, out, stream);
}

// ---------------------------------------------------------------- TMA gather4
//
// The same measurement with the rows fetched by the tensor memory accelerator:
// one cp.async.bulk.tensor .tile::gather4 brings four rows (named by their row
// coordinates, box one row high) of a 2-D tensor map over the row set into
// shared memory and signals an mbarrier; one lane per warp issues it, kStages
// gathers ahead, and the warp adds the rows from shared memory. Each wait on
// an mbarrier is bounded: when it runs out the kernel sets an error word,
// waits (bounded again) for its own copies still in flight, and stops.
namespace cbtbe {
namespace {

constexpr int kTmaStages = 8;         // gathers in flight per warp
constexpr int kTmaWarps = 8;          // warps per block
constexpr uint32_t kSpinLimit = 1u << 22;  // polls of one mbarrier before giving up

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arm(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool mbar_try(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait for the phase `parity` of `bar` to complete.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
    for (uint32_t i = 0; i < kSpinLimit; ++i)
        if (mbar_try(bar, parity)) return true;
    return false;
}
__device__ __forceinline__ void tma_gather4(void* dst, const CUtensorMap* map, int32_t col, int32_t r0, int32_t r1,
                                            int32_t r2, int32_t r3, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile::gather4.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4, %5, %6}], [%7];\n" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(col), "r"(r0), "r"(r1), "r"(r2), "r"(r3), "r"(smem_u32(bar))
        : "memory");
}

template <int RB>
__global__ void __launch_bounds__(kTmaWarps * 32) gather4_ceiling_kernel(const __grid_constant__ CUtensorMap map,
                                                                        const uint32_t* __restrict__ idx,
                                                                        int64_t num_rows, int64_t n,
                                                                        float* __restrict__ out, int* err) {
    constexpr int kSlot = 4 * RB;                 // bytes of one gather (4 rows)
    constexpr int kVec = kSlot / 16 / 32;         // 16-byte vectors per lane per gather
    extern __shared__ unsigned char dyn[];
    unsigned char* base = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(dyn) + 1023) & ~uintptr_t(1023));
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    unsigned char* ring = base + static_cast<size_t>(w) * kTmaStages * kSlot;
    uint64_t* bars = reinterpret_cast<uint64_t*>(base + static_cast<size_t>(kTmaWarps) * kTmaStages * kSlot) +
                     w * kTmaStages;
    if (lane == 0)
        for (int s = 0; s < kTmaStages; ++s) mbar_init(bars + s, 1);
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    __syncwarp();
    const int64_t batches = (n + 31) / 32;
    const int64_t wg = static_cast<int64_t>(blockIdx.x) * kTmaWarps + w, nw = static_cast<int64_t>(gridDim.x) * kTmaWarps;
    const int64_t my_batches = wg < batches ? (batches - wg + nw - 1) / nw : 0;
    const int64_t total = my_batches * 8;         // gathers of this warp (8 per batch of 32)
    // The rows of the warp's gathers: lane l holds item l of the batch being
    // issued (cur) and of the next one (nxt), loaded a batch ahead; the issuing
    // lane takes a gather's four rows by shuffle.
    auto batch_rows = [&](int64_t kb) -> int32_t {
        const int64_t q = (wg + kb * nw) * 32 + lane;
        if (kb >= my_batches || q >= n) return static_cast<int32_t>(num_rows);  // a zero-filled row
        const uint32_t r = __ldg(idx + q);
        return r < num_rows ? static_cast<int32_t>(r) : 0;
    };
    int32_t cur = batch_rows(0), nxt = batch_rows(1);
    int64_t issued = 0;
    auto issue = [&]() {  // the whole warp; lane 0 issues
        if ((issued & 7) == 0 && issued > 0) {
            cur = nxt;
            nxt = batch_rows((issued >> 3) + 1);
        }
        const int b4 = static_cast<int>(issued & 7) * 4;
        const int32_t r0 = __shfl_sync(kFull, cur, b4), r1 = __shfl_sync(kFull, cur, b4 + 1);
        const int32_t r2 = __shfl_sync(kFull, cur, b4 + 2), r3 = __shfl_sync(kFull, cur, b4 + 3);
        if (lane == 0) {
            const int s = static_cast<int>(issued % kTmaStages);
            asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
            mbar_arm(bars + s, kSlot);
            tma_gather4(ring + s * kSlot, &map, 0, r0, r1, r2, r3, bars + s);
        }
        ++issued;
    };
    while (issued < total && issued < kTmaStages) issue();
    float acc = 0.f;
    bool failed = false;
    for (int64_t k = 0; k < total; ++k) {
        const int s = static_cast<int>(k % kTmaStages);
        const uint32_t parity = static_cast<uint32_t>((k / kTmaStages) & 1);
        const bool ok = mbar_wait(bars + s, parity);
        if (!__all_sync(kFull, ok)) {
            failed = true;
            break;
        }
        const uint4* v = reinterpret_cast<const uint4*>(ring + s * kSlot);
#pragma unroll
        for (int x = 0; x < kVec; ++x) {
            const uint4 y = v[lane + 32 * x];
            acc += (__uint_as_float(y.x) + __uint_as_float(y.y)) + (__uint_as_float(y.z) + __uint_as_float(y.w));
        }
        if ((k & 7) == 7) {  // a batch of 32 items is complete
            float t = acc;
#pragma unroll
            for (int off = 16; off >= 1; off >>= 1) t += __shfl_xor_sync(kFull, t, off);
            if (lane == 0) out[wg + (k >> 3) * nw] = t;
            acc = 0.f;
        }
        __syncwarp();  // every lane has read slot s before it is refilled
        if (issued < total) issue();
    }
    if (failed) {
        if (lane == 0) atomicExch(err, CB_ERR_TIMEOUT);
        // copies still in flight land before the block's shared memory goes away
        for (int64_t k = 0; k < issued; ++k) {
            const int s = static_cast<int>(k % kTmaStages);
            if (!mbar_wait(bars + s, static_cast<uint32_t>((k / kTmaStages) & 1))) break;
        }
    }
}

template <int RB>
size_t gather4_smem() {
    return static_cast<size_t>(kTmaWarps) * kTmaStages * 4 * RB + kTmaWarps * kTmaStages * sizeof(uint64_t) + 1024;
}

template <int RB>
cb_status launch4(const CUtensorMap& map, int64_t num_rows, const uint32_t* idx, int64_t n, float* out, int* err,
                  cudaStream_t s) {
    int dev = 0, sms = 1;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
        cudaGetLastError();
        return CB_ERR_CUDA;
    }
    const size_t smem = gather4_smem<RB>();
    if (cudaFuncSetAttribute(gather4_ceiling_kernel<RB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem)) != cudaSuccess) {
        cudaGetLastError();
        return CB_ERR_CUDA;
    }
    int per_sm = 1;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gather4_ceiling_kernel<RB>, kTmaWarps * 32, smem) !=
            cudaSuccess || per_sm < 1)
        per_sm = 1;
    const int64_t batches = (n + 31) / 32;
    const int64_t need = (batches + kTmaWarps - 1) / kTmaWarps;
    const int grid = static_cast<int>(need < per_sm * sms ? (need > 0 ? need : 1) : per_sm * sms);
    gather4_ceiling_kernel<RB><<<grid, kTmaWarps * 32, smem, s>>>(map, idx, num_rows, n, out, err);
    return cudaGetLastError() == cudaSuccess ? CB_OK : CB_ERR_CUDA;
}

}  // namespace
}  // namespace cbtbe

extern "C" cb_status cb_gather_ceiling_tma(const void* rows, int64_t num_rows, int32_t row_bytes,
                                           const uint32_t* indices, int64_t num_indices, float* out,
                                           int* error, cudaStream_t stream) {
    using namespace cbtbe;
    if (!rows || num_rows <= 0 || num_rows >= (int64_t(1) << 31) || num_indices < 0 || !error ||
        (num_indices > 0 && (!indices || !out)) || (reinterpret_cast<uintptr_t>(rows) & 15u))
        return CB_ERR_INVALID_ARG;
    if (row_bytes != 256 && row_bytes != 512) return CB_ERR_INVALID_ARG;
    if (num_indices == 0) return CB_OK;
    static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    if (!encode) {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
                cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) {
            cudaGetLastError();
            return CB_ERR_CUDA;
        }
        encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    // The row set as a 2-D fp32 tensor [num_rows, row_bytes / 4]; the box is
    // one whole row (one row high, as .tile::gather4 requires).
    CUtensorMap map;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(row_bytes / 4), static_cast<cuuint64_t>(num_rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(row_bytes)};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(row_bytes / 4), 1};
    const cuuint32_t estr[2] = {1, 1};
    if (encode(&map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(rows), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return CB_ERR_INVALID_ARG;
    return row_bytes == 256 ? launch4<256>(map, num_rows, indices, num_indices, out, error, stream)
                            : launch4<512>(map, num_rows, indices, num_indices, out, error, stream);
}
