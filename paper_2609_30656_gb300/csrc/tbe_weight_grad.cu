// tbe_weight_grad.cu -- gradient of the pooled output with respect to the
// per-sample weights. The pooled bag (Sec. IV.A.2 sparse_arch lookups) is
// linear in each weight, so for an upstream gradient grad_out
//
//   grad_w[i] = s_b * sum_j grad_out[b, Doff_t + j] * E_t[indices[i], j]
//
// (s_b = 1/L for mean pooling, 1 for sum), whatever the weights are: one dot
// product of the lookup's table row with its bag's grad_out slice.
//
// One warp per chunk of lookup positions (the forward's chunk plan). Each lane
// finds the bag of one position of a 32-position batch by bisection over a
// window of bag ends; then G = 32 / V lookups per warp step (V lanes per stored
// row, 16 bytes each), several steps' loads in flight, a dot product per lane
// and a butterfly over the row's lanes. Consecutive lookups of one bag read the
// same grad_out slice, which L1 serves. grad_out is fp32, or fp16 / bf16 when
// the handle's output is (mixed precision). The dot products are summed in a
// fixed order (deterministic).
#include "tbe_internal.cuh"
#include "tbe_launch.h"

namespace cbtbe {
namespace {

constexpr int kWgradSteps = 4;  // warp steps whose loads are issued together

// Four grad_out values at g (fp32, or fp16 / bf16 with mixed precision), widened.
__device__ __forceinline__ float4 load_go4(const char* g, int go_dtype) {
    if (go_dtype == CB_F32) return __ldg(reinterpret_cast<const float4*>(g));
    const uint2 w = __ldg(reinterpret_cast<const uint2*>(g));
    if (go_dtype == CB_BF16)
        return make_float4(__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xffff0000u),
                           __uint_as_float(w.y << 16), __uint_as_float(w.y & 0xffff0000u));
    __half2 a, b;
    memcpy(&a, &w.x, 4);
    memcpy(&b, &w.y, 4);
    const float2 fa = __half22float2(a), fb = __half22float2(b);
    return make_float4(fa.x, fa.y, fb.x, fb.y);
}

// <row vector x, the E grad_out values at g>, g in bytes of the grad_out type.
template <int DT>
__device__ __forceinline__ float dot_row(const uint4& x, const char* g, int go_dtype) {
    constexpr int E = Storage<DT>::kElems;
    float f[E];
    unpack<DT>(x, f);
    const int step = go_dtype == CB_F32 ? 16 : 8;
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < E / 4; ++k) {
        const float4 q = load_go4(g + k * step, go_dtype);
        acc = fmaf(q.x, f[4 * k], acc);
        acc = fmaf(q.y, f[4 * k + 1], acc);
        acc = fmaf(q.z, f[4 * k + 2], acc);
        acc = fmaf(q.w, f[4 * k + 3], acc);
    }
    return acc;
}

// GC > 0: rows of exactly V = 32 / GC vectors (one per lane), GC lookups per
// warp step. GC == 0: any row size, one lookup per step, each lane taking
// vectors lane, lane + 32, ... of the row.
template <int DT, int GC>
__global__ void __launch_bounds__(kWarpThreads) weight_grad_kernel(const __grid_constant__ Problem P,
                                                                   const __grid_constant__ Plan Q,
                                                                   const void* grad_out, float* grad_w,
                                                                   int cls) {
    constexpr int E = Storage<DT>::kElems;
    constexpr int G = GC > 0 ? GC : 1;
    constexpr int V = 32 / G;
    const int lane = threadIdx.x & 31;
    const int g = lane / V, v = lane - g * V;
    const int64_t cb = Q.class_chunk_base[cls];
    const int64_t ce = min64(Q.class_chunk_base[cls + 1], Q.max_chunks);
    for (int64_t j = first_chunk(Q, cls, cb, lane); j < ce;) {
        const int64_t nxt = fetch_next_chunk(Q, cls, cb, lane);
        const Chunk ch = Q.chunks[j];
        const int t = ch.table;
        const TableDev& td = P.tables[t];
        const uint4* rows = static_cast<const uint4*>(td.data);
        const int nvec = td.row_vecs;
        const int64_t k0 = ch.k0, k1 = ch.k0 + (ch.len & 0x7fffffffu);
        const int64_t bag_lo = static_cast<int64_t>(t) * P.B, bag_hi = bag_lo + P.B;
        const int eb = dtype_bytes(P.out_dtype);
        const char* go_base = static_cast<const char*>(grad_out) + static_cast<int64_t>(td.doff) * eb;
        BagWindow W = bag_window(P, ch.first, bag_hi, lane);
        for (int64_t base = k0; base < k1; base += 32) {
            const int64_t q = base + lane;
            const bool valid = q < k1;
            int64_t my_bag, my_s, my_e;
            find_bag(P, W, q, valid, lane, my_bag, my_s, my_e);
            // Per position: row (kInvalid = contributes nothing), bag row offset, s_b.
            uint32_t my_a = kInvalid;
            int64_t my_go = 0;
            float my_sc = 0.f;
            if (valid) {
                if (my_bag >= bag_hi) {  // only reachable with malformed offsets
                    set_error(P.error, CB_ERR_BAD_OFFSETS);
                    my_bag = bag_hi - 1;
                }
                const int64_t r = load_index(P.indices, q, P.is32);
                if (r < 0 || r >= td.rows) set_error(P.error, CB_ERR_INDEX_OOB);
                else my_a = static_cast<uint32_t>(r);
                my_go = (my_bag - bag_lo) * P.sum_d;
                my_sc = (P.mean && my_e > my_s) ? 1.f / static_cast<float>(my_e - my_s) : 1.f;
            }
            const int nb = static_cast<int>(min64(32, k1 - base));
            for (int i0 = 0; i0 < nb; i0 += G * kWgradSteps) {
                float dot[kWgradSteps];
#pragma unroll
                for (int u = 0; u < kWgradSteps; ++u) {
                    const int i = i0 + u * G + g;
                    const uint32_t a = __shfl_sync(kFull, my_a, i & 31);
                    const int64_t go = __shfl_sync(kFull, my_go, i & 31);
                    dot[u] = 0.f;
                    if (i >= nb || a == kInvalid) continue;
                    const uint4* rp = rows + static_cast<int64_t>(a) * nvec;
                    const char* gp = go_base + go * eb;
                    if (GC > 0) {
                        dot[u] = dot_row<DT>(__ldg(rp + v), gp + v * E * eb, P.out_dtype);
                    } else {
                        for (int vec = v; vec < nvec; vec += 32)
                            dot[u] += dot_row<DT>(__ldg(rp + vec), gp + vec * E * eb, P.out_dtype);
                    }
                }
#pragma unroll
                for (int u = 0; u < kWgradSteps; ++u) {
#pragma unroll
                    for (int off = V / 2; off >= 1; off >>= 1) dot[u] += __shfl_xor_sync(kFull, dot[u], off);
                    const int i = i0 + u * G + g;
                    const float sc = __shfl_sync(kFull, my_sc, i & 31);
                    if (v == 0 && i < nb) grad_w[base + i] = sc * dot[u];
                }
            }
        }
        j = __shfl_sync(kFull, nxt, 0);
    }
}

template <int DT, int GC>
void launch_one(const Problem& P, const Plan& Q, const void* go, float* gw, int cls, int64_t chunk_bound,
                int num_sms, cudaStream_t s) {
    static int per_sm = -1;
    if (per_sm < 0 && (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, weight_grad_kernel<DT, GC>,
                                                                     kWarpThreads, 0) != cudaSuccess ||
                       per_sm < 1))
        per_sm = 1;
    const int64_t need = (chunk_bound + (kWarpThreads / 32) - 1) / (kWarpThreads / 32);
    const int grid = static_cast<int>(max64(1, min64(need, static_cast<int64_t>(per_sm) * num_sms)));
    weight_grad_kernel<DT, GC><<<grid, kWarpThreads, 0, s>>>(P, Q, go, gw, cls);
}

template <int DT>
void launch_dtype(const Problem& P, const Plan& Q, const void* go, float* gw, int cls, int gc,
                  int64_t chunk_bound, int num_sms, cudaStream_t s) {
    switch (gc) {
        case 1: launch_one<DT, 1>(P, Q, go, gw, cls, chunk_bound, num_sms, s); break;
        case 2: launch_one<DT, 2>(P, Q, go, gw, cls, chunk_bound, num_sms, s); break;
        case 4: launch_one<DT, 4>(P, Q, go, gw, cls, chunk_bound, num_sms, s); break;
        case 8: launch_one<DT, 8>(P, Q, go, gw, cls, chunk_bound, num_sms, s); break;
        default: launch_one<DT, 0>(P, Q, go, gw, cls, chunk_bound, num_sms, s); break;
    }
}

}  // namespace

void launch_weight_grad(const Problem& P, const Plan& Q, const void* grad_out, float* grad_w, int cls,
                        int dtype, int gc, int64_t chunk_bound, int num_sms, cudaStream_t s) {
    if (dtype == CB_F32) launch_dtype<CB_F32>(P, Q, grad_out, grad_w, cls, gc, chunk_bound, num_sms, s);
    else if (dtype == CB_F16) launch_dtype<CB_F16>(P, Q, grad_out, grad_w, cls, gc, chunk_bound, num_sms, s);
    else launch_dtype<CB_BF16>(P, Q, grad_out, grad_w, cls, gc, chunk_bound, num_sms, s);
}

}  // namespace cbtbe
