// fm_interaction.cu -- the factorization-machine cross term on the pooled
// embeddings and its gradient: the inter_arch.fm step that follows the
// lookups in the paper's DeepFM-based model (Sec. IV.A.2, where it is
// bandwidth-bound: a few element-wise and reduction passes over the pooled
// rows). With each table's pooled row as one field embedding,
// v_bt = y[b, t*D : (t+1)*D], the second-order term of the factorization
// machine (Rendle, 2010, cited by the paper) is
//
//   fm[b] = sum_{t < u} <v_bt, v_bu> = 1/2 sum_j [(sum_t v_btj)^2 - sum_t v_btj^2]
//
// and, for an upstream gradient g[b],
//
//   grad_y[b, t*D + j] = g[b] * (sum_u v_buj - v_btj).
//
// The forward runs one warp per sample: the warp streams the sample's T*D
// values with 16-byte loads and keeps per-column sums and sums of squares in
// registers, reading every value once. The backward runs one block per sample
// when the row fits the block's registers (up to 4096 16-byte vectors): the row
// is loaded once, the column sums meet in shared memory, and the gradient row is
// written from registers; other shapes take a warp per sample that reads the
// row twice. Sums are taken in a fixed order, so results are deterministic.
#include <cstdint>
#include <cuda_runtime.h>

#include "cb_tbe.h"

namespace cbtbe {
namespace {

constexpr int kFmThreads = 256;

__device__ __forceinline__ void add4(float4& a, const float4& x) {
    a.x += x.x;
    a.y += x.y;
    a.z += x.z;
    a.w += x.w;
}
__device__ __forceinline__ void fma4(float4& a, const float4& x) {
    a.x = fmaf(x.x, x.x, a.x);
    a.y = fmaf(x.y, x.y, a.y);
    a.z = fmaf(x.z, x.z, a.z);
    a.w = fmaf(x.w, x.w, a.w);
}
__device__ __forceinline__ float4 shfl_xor4(const float4& a, int off) {
    return make_float4(__shfl_xor_sync(0xffffffffu, a.x, off), __shfl_xor_sync(0xffffffffu, a.y, off),
                       __shfl_xor_sync(0xffffffffu, a.z, off), __shfl_xor_sync(0xffffffffu, a.w, off));
}

// Field layout over a warp, with nv = D / 4 vectors per field: G = 32 / nv
// fields side by side per step when nv divides 32 (D <= 128, M = 1); otherwise
// one field per step, lane l owning vector columns l + 32 m for m < M.
template <int G, int M>
struct FieldMap {
    int g, c;  // field group of this lane, its first vector column
    int nv;
    __device__ FieldMap(int lane, int nv_) : nv(nv_) {
        g = G > 1 ? lane / (32 / G) : 0;
        c = G > 1 ? lane - g * (32 / G) : lane;
    }
    __device__ bool live(int m) const { return c + 32 * m < nv; }
    __device__ int64_t at(int t, int m) const { return static_cast<int64_t>(t) * nv + c + 32 * m; }
};

// Column sums s (and sums of squares q) of one sample, combined over the G
// field groups so every group holds the totals of its columns.
template <int G, int M, bool SQUARES>
__device__ __forceinline__ void column_sums(const float4* row, int T, const FieldMap<G, M>& f,
                                            float4 (&s)[M], float4 (&q)[M]) {
#pragma unroll
    for (int m = 0; m < M; ++m) s[m] = q[m] = make_float4(0.f, 0.f, 0.f, 0.f);
    int t = f.g;
    for (; t + 3 * G < T; t += 4 * G) {
        float4 x[4][M];
#pragma unroll
        for (int k = 0; k < 4; ++k)
#pragma unroll
            for (int m = 0; m < M; ++m)
                x[k][m] = f.live(m) ? __ldg(row + f.at(t + k * G, m)) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int k = 0; k < 4; ++k)
#pragma unroll
            for (int m = 0; m < M; ++m) {
                add4(s[m], x[k][m]);
                if (SQUARES) fma4(q[m], x[k][m]);
            }
    }
    for (; t < T; t += G) {
#pragma unroll
        for (int m = 0; m < M; ++m) {
            const float4 x = f.live(m) ? __ldg(row + f.at(t, m)) : make_float4(0.f, 0.f, 0.f, 0.f);
            add4(s[m], x);
            if (SQUARES) fma4(q[m], x);
        }
    }
#pragma unroll
    for (int off = 32 / G; off < 32; off <<= 1)
#pragma unroll
        for (int m = 0; m < M; ++m) {
            add4(s[m], shfl_xor4(s[m], off));
            if (SQUARES) add4(q[m], shfl_xor4(q[m], off));
        }
}

template <int G, int M>
__global__ void __launch_bounds__(kFmThreads) fm_forward_kernel(const float* __restrict__ y, int B, int T,
                                                                int nv, int64_t stride,
                                                                float* __restrict__ out) {
    const int lane = threadIdx.x & 31;
    const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    const FieldMap<G, M> f(lane, nv);
    for (int64_t b = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5; b < B;
         b += nwarps) {
        float4 s[M], q[M];
        column_sums<G, M, true>(reinterpret_cast<const float4*>(y + b * stride), T, f, s, q);
        float part = 0.f;
        if (f.g == 0) {
#pragma unroll
            for (int m = 0; m < M; ++m)
                if (f.live(m))
                    part += (fmaf(s[m].x, s[m].x, -q[m].x) + fmaf(s[m].y, s[m].y, -q[m].y)) +
                            (fmaf(s[m].z, s[m].z, -q[m].z) + fmaf(s[m].w, s[m].w, -q[m].w));
        }
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) part += __shfl_xor_sync(0xffffffffu, part, off);
        if (lane == 0) out[b] = 0.5f * part;
    }
}

template <int G, int M>
__global__ void __launch_bounds__(kFmThreads) fm_backward_kernel(const float* __restrict__ y,
                                                                 const float* __restrict__ grad_fm, int B,
                                                                 int T, int nv, int64_t stride,
                                                                 float* __restrict__ grad_y) {
    const int lane = threadIdx.x & 31;
    const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    const FieldMap<G, M> f(lane, nv);
    for (int64_t b = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5; b < B;
         b += nwarps) {
        const float4* row = reinterpret_cast<const float4*>(y + b * stride);
        float4* dst = reinterpret_cast<float4*>(grad_y + b * stride);
        float4 s[M], q[M];
        column_sums<G, M, false>(row, T, f, s, q);
        const float gb = __ldg(grad_fm + b);
        for (int t = f.g; t < T; t += G) {
#pragma unroll
            for (int m = 0; m < M; ++m) {
                if (!f.live(m)) continue;
                const float4 x = row[f.at(t, m)];
                dst[f.at(t, m)] = make_float4(gb * (s[m].x - x.x), gb * (s[m].y - x.y), gb * (s[m].z - x.z),
                                              gb * (s[m].w - x.w));
            }
        }
    }
}

// Backward with one block per sample when 256 threads tile the sample's row:
// nv divides 256 (so thread i always owns vector column i % nv) and the row
// has at most 256 * K vectors. The row stays in registers between the column
// sums and the gradient, so it is read from memory once.
constexpr int kRowThreads = 256;

template <int K>
__global__ void __launch_bounds__(kRowThreads) fm_backward_rows_kernel(const float* __restrict__ y,
                                                                       const float* __restrict__ grad_fm,
                                                                       int B, int T, int nv, int64_t stride,
                                                                       float* __restrict__ grad_y) {
    __shared__ float4 part[kRowThreads];
    const int i = threadIdx.x;
    const int c = i % nv, r = i / nv, R = kRowThreads / nv;
    const int nvec = T * nv;  // vector k of the row is field k / nv, column k % nv
    for (int64_t b = blockIdx.x; b < B; b += gridDim.x) {
        const float4* row = reinterpret_cast<const float4*>(y + b * stride);
        float4 x[K];
        float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int j = 0; j < K; ++j) {
            const int k = i + kRowThreads * j;
            x[j] = k < nvec ? __ldg(row + k) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int j = 0; j < K; ++j) add4(s, x[j]);
        part[i] = s;
        __syncthreads();
        if (r == 0) {  // column c: the R partial sums in a fixed order
            float4 S = part[c];
            for (int q = 1; q < R; ++q) add4(S, part[q * nv + c]);
            part[c] = S;
        }
        __syncthreads();
        const float4 S = part[c];
        const float gb = __ldg(grad_fm + b);
        float4* dst = reinterpret_cast<float4*>(grad_y + b * stride);
#pragma unroll
        for (int j = 0; j < K; ++j) {
            const int k = i + kRowThreads * j;
            if (k < nvec)
                dst[k] = make_float4(gb * (S.x - x[j].x), gb * (S.y - x[j].y), gb * (S.z - x[j].z),
                                     gb * (S.w - x[j].w));
        }
        __syncthreads();  // `part` is reused by the next sample
    }
}

int sm_count() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
        return 1;
    return n;
}

// Warps per SM the grid asks for: enough 16-byte loads in flight to cover HBM
// latency; samples beyond the grid are taken in a grid-stride loop.
constexpr int kFmBlocksPerSm = 8;

template <int G, int M>
void launch_fm(bool backward, const float* y, const float* grad_fm, int B, int T, int nv,
               int64_t stride, float* out, cudaStream_t s) {
    const int64_t warps_per_block = kFmThreads / 32;
    const int64_t need = (static_cast<int64_t>(B) + warps_per_block - 1) / warps_per_block;
    const int grid = static_cast<int>(need < int64_t(sm_count()) * kFmBlocksPerSm ? need
                                                                                   : int64_t(sm_count()) * kFmBlocksPerSm);
    if (backward)
        fm_backward_kernel<G, M><<<grid, kFmThreads, 0, s>>>(y, grad_fm, B, T, nv, stride, out);
    else
        fm_forward_kernel<G, M><<<grid, kFmThreads, 0, s>>>(y, B, T, nv, stride, out);
}

cb_status fm_call(bool backward, const float* y, const float* grad_fm, int32_t batch, int32_t num_fields,
                  int32_t dim, int64_t row_stride, float* out, cudaStream_t stream) {
    if (batch < 0 || num_fields < 1 || dim < 4 || dim > 512 || (dim & 3) ||
        row_stride < static_cast<int64_t>(num_fields) * dim || (row_stride & 3))
        return CB_ERR_INVALID_ARG;
    if (batch > 0 && (!y || !out || (backward && !grad_fm))) return CB_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(y) & 15u) || (backward && (reinterpret_cast<uintptr_t>(out) & 15u)))
        return CB_ERR_INVALID_ARG;
    if (batch == 0) return CB_OK;
    cudaGetLastError();  // an earlier, unrelated failure is not this call's
    const int nv = dim / 4;
    const int64_t nvec = static_cast<int64_t>(num_fields) * nv;
    if (backward && kRowThreads % nv == 0 && nvec <= 16 * kRowThreads) {
        const int k = nvec <= 4 * kRowThreads ? 4 : (nvec <= 8 * kRowThreads ? 8 : 16);
        const int per_sm = k == 16 ? 2 : 4;
        const int grid = static_cast<int>(batch < sm_count() * per_sm * 4 ? batch : sm_count() * per_sm * 4);
        if (k == 4)
            fm_backward_rows_kernel<4><<<grid, kRowThreads, 0, stream>>>(y, grad_fm, batch, num_fields, nv,
                                                                        row_stride, out);
        else if (k == 8)
            fm_backward_rows_kernel<8><<<grid, kRowThreads, 0, stream>>>(y, grad_fm, batch, num_fields, nv,
                                                                        row_stride, out);
        else
            fm_backward_rows_kernel<16><<<grid, kRowThreads, 0, stream>>>(y, grad_fm, batch, num_fields, nv,
                                                                         row_stride, out);
        return cudaGetLastError() == cudaSuccess ? CB_OK : CB_ERR_CUDA;
    }
    if (nv <= 32 && 32 % nv == 0) {
        switch (32 / nv) {
            case 1: launch_fm<1, 1>(backward, y, grad_fm, batch, num_fields, nv, row_stride, out, stream); break;
            case 2: launch_fm<2, 1>(backward, y, grad_fm, batch, num_fields, nv, row_stride, out, stream); break;
            case 4: launch_fm<4, 1>(backward, y, grad_fm, batch, num_fields, nv, row_stride, out, stream); break;
            case 8: launch_fm<8, 1>(backward, y, grad_fm, batch, num_fields, nv, row_stride, out, stream); break;
            case 16: launch_fm<16, 1>(backward, y, grad_fm, batch, num_fields, nv, row_stride, out, stream); break;
            default: launch_fm<32, 1>(backward, y, grad_fm, batch, num_fields, nv, row_stride, out, stream); break;
        }
    } else {
        switch ((nv + 31) / 32) {
            case 1: launch_fm<1, 1>(backward, y, grad_fm, batch, num_fields, nv, row_stride, out, stream); break;
            case 2: launch_fm<1, 2>(backward, y, grad_fm, batch, num_fields, nv, row_stride, out, stream); break;
            case 3: launch_fm<1, 3>(backward, y, grad_fm, batch, num_fields, nv, row_stride, out, stream); break;
            default: launch_fm<1, 4>(backward, y, grad_fm, batch, num_fields, nv, row_stride, out, stream); break;
        }
    }
    return cudaGetLastError() == cudaSuccess ? CB_OK : CB_ERR_CUDA;
}

}  // namespace
}  // namespace cbtbe

extern "C" cb_status cb_fm_forward(const float* y, int32_t batch, int32_t num_fields, int32_t dim,
                                   int64_t row_stride, float* out, cudaStream_t stream) {
    return cbtbe::fm_call(false, y, nullptr, batch, num_fields, dim, row_stride, out, stream);
}

extern "C" cb_status cb_fm_backward(const float* y, const float* grad_fm, int32_t batch,
                                    int32_t num_fields, int32_t dim, int64_t row_stride, float* grad_y,
                                    cudaStream_t stream) {
    return cbtbe::fm_call(true, y, grad_fm, batch, num_fields, dim, row_stride, grad_y, stream);
}
