// kjt_replicate.cu -- the batch-size preprocessor of Component Benchmark
// (Sec. III): a small captured batch of jagged lookups is replicated to the
// production batch size, which keeps the input distribution the lookup sees.
// For T tables and a key-major batch of B bags per table, the output has
// F * B bags per table, and bag r * B + b of table t is bag b of table t:
//
//   out_offsets[t*F*B + r*B + b] = F * off[t*B] + r * n_t + (off[t*B + b] - off[t*B])
//   out_indices[F * off[t*B] + r * n_t + i] = indices[off[t*B] + i]   (i < n_t)
//
// with n_t = off[(t+1)*B] - off[t*B]. Two grid-stride kernels, one over the
// output offsets and one over the output lookups (the table of a lookup by
// bisection over the T + 1 table starts). Offsets are clamped into [0, n] and
// made monotone per table first, so any input stays in bounds.
#include <cstdint>
#include <cuda_runtime.h>

#include "cb_tbe.h"

namespace cbtbe {
namespace {

template <typename I>
__device__ __forceinline__ int64_t off_at(const I* off, int64_t k, int64_t n) {
    const int64_t v = static_cast<int64_t>(off[k]);
    return v < 0 ? 0 : (v > n ? n : v);
}

template <typename I>
__global__ void replicate_offsets_kernel(const I* off, int32_t T, int32_t B, int64_t n, int32_t F,
                                         I* out) {
    const int64_t total = static_cast<int64_t>(T) * F * B;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t k = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; k <= total; k += stride) {
        if (k == total) {
            out[k] = static_cast<I>(static_cast<int64_t>(F) * off_at(off, static_cast<int64_t>(T) * B, n));
            continue;
        }
        const int64_t t = k / (static_cast<int64_t>(F) * B);
        const int64_t rem = k - t * F * B;
        const int64_t r = rem / B, b = rem - r * B;
        const int64_t s = off_at(off, t * B, n);
        const int64_t e = off_at(off, (t + 1) * B, n) < s ? s : off_at(off, (t + 1) * B, n);
        int64_t ob = off_at(off, t * B + b, n);
        ob = ob < s ? s : (ob > e ? e : ob);
        out[k] = static_cast<I>(static_cast<int64_t>(F) * s + r * (e - s) + (ob - s));
    }
}

template <typename I>
__global__ void replicate_lookups_kernel(const I* ind, const I* off, const float* w, int32_t T, int32_t B,
                                         int64_t n, int32_t F, I* out_ind, float* out_w) {
    const int64_t total = static_cast<int64_t>(F) * off_at(off, static_cast<int64_t>(T) * B, n);
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t q = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; q < total; q += stride) {
        // largest t with F * off[t*B] <= q
        int lo = 0, hi = T;
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (static_cast<int64_t>(F) * off_at(off, static_cast<int64_t>(mid) * B, n) <= q) lo = mid;
            else hi = mid;
        }
        const int64_t s = off_at(off, static_cast<int64_t>(lo) * B, n);
        const int64_t e = off_at(off, static_cast<int64_t>(lo + 1) * B, n);
        const int64_t nt = e > s ? e - s : 0;
        const int64_t rel = q - static_cast<int64_t>(F) * s;
        if (nt == 0 || rel < 0 || rel >= static_cast<int64_t>(F) * nt) continue;  // only with bad offsets
        const int64_t src = s + rel % nt;
        out_ind[q] = ind[src];
        if (w) out_w[q] = w[src];
    }
}

int grid_for(int64_t work) {
    int dev = 0, sms = 1;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t blocks = (work + 255) / 256;
    const int64_t cap = static_cast<int64_t>(sms > 0 ? sms : 1) * 16;
    return static_cast<int>(blocks < 1 ? 1 : (blocks < cap ? blocks : cap));
}

template <typename I>
void launch(const void* ind, const void* off, const float* w, int32_t T, int32_t B, int64_t n, int32_t F,
            void* out_ind, void* out_off, float* out_w, cudaStream_t s) {
    const int64_t bags = static_cast<int64_t>(T) * F * B + 1;
    replicate_offsets_kernel<I><<<grid_for(bags), 256, 0, s>>>(static_cast<const I*>(off), T, B, n, F,
                                                              static_cast<I*>(out_off));
    if (n > 0)
        replicate_lookups_kernel<I><<<grid_for(static_cast<int64_t>(F) * n), 256, 0, s>>>(
            static_cast<const I*>(ind), static_cast<const I*>(off), w, T, B, n, F, static_cast<I*>(out_ind),
            out_w);
}

}  // namespace
}  // namespace cbtbe

extern "C" cb_status cb_kjt_replicate(const void* indices, const void* offsets, const float* per_sample_weights,
                                      cb_index_dtype idx_dtype, int32_t num_tables, int32_t batch,
                                      int64_t num_indices, int32_t factor, void* out_indices,
                                      void* out_offsets, float* out_weights, cudaStream_t stream) {
    if (num_tables < 1 || batch < 0 || num_indices < 0 || factor < 1 || !offsets || !out_offsets)
        return CB_ERR_INVALID_ARG;
    if (idx_dtype != CB_I32 && idx_dtype != CB_I64) return CB_ERR_INVALID_ARG;
    if (num_indices > 0 && (!indices || !out_indices)) return CB_ERR_INVALID_ARG;
    if (per_sample_weights && num_indices > 0 && !out_weights) return CB_ERR_INVALID_ARG;
    const int64_t nn = static_cast<int64_t>(factor) * num_indices;
    const int64_t bags = static_cast<int64_t>(num_tables) * factor * batch;
    if (bags >= (int64_t(1) << 31) || (idx_dtype == CB_I32 && nn > INT32_MAX)) return CB_ERR_INVALID_ARG;
    cudaGetLastError();
    if (idx_dtype == CB_I64)
        cbtbe::launch<long long>(indices, offsets, per_sample_weights, num_tables, batch, num_indices, factor,
                                 out_indices, out_offsets, out_weights, stream);
    else
        cbtbe::launch<int>(indices, offsets, per_sample_weights, num_tables, batch, num_indices, factor,
                           out_indices, out_offsets, out_weights, stream);
    return cudaGetLastError() == cudaSuccess ? CB_OK : CB_ERR_CUDA;
}
