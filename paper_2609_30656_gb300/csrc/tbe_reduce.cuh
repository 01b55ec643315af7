// tbe_reduce.cuh -- the backward segmented reduce (runs of equal sorted row
// ids; per run the coefficient-weighted sum of the gathered grad_out slices,
// the de-duplicated adjoint of the pooled bag of Sec. IV.A.2), and the
// optimizer step that can be fused where a run's sum ends. Included by
// tbe_backward.cu (gradient output) and tbe_backward_apply.cu (fused step).
#pragma once

#include <cuda_bf16.h>

#include "tbe_internal.cuh"
#include "tbe_launch.h"

// The reduce with the optimizer step fused carries more state (the table row
// and its update), so it spilled at 3 blocks with 8 rows; measured on cfg5
// (fused SGD / Adagrad ms): 8 rows at 3 blocks 14.46 / 17.24, 4 at 4 13.25 /
// 15.47, 4 at 5 13.00 / 15.05, 2 at 5 12.93 / 14.83, 2 at 6 13.22 / 14.88,
// 1 at 5 13.73 / 15.67.
#ifndef CB_REDUCE_APPLY_ROWS
#define CB_REDUCE_APPLY_ROWS 2  // rows in flight per lane with the optimizer step fused
#endif
#ifndef CB_REDUCE_HALF_ROWS
#define CB_REDUCE_HALF_ROWS 4  // rows in flight per lane for fp16 / bf16 grad_out
#endif
#ifndef CB_REDUCE_HALF_FAST_BATCH
#define CB_REDUCE_HALF_FAST_BATCH 1  // fp16 / bf16 grad_out: unrolled path for batches with no run end
#endif

namespace cbtbe {

template <class KernelT>
inline int occupancy_grid(KernelT kernel, int threads, int num_sms) {
    int per_sm = 1;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, 0) != cudaSuccess ||
        per_sm < 1)
        per_sm = 1;
    return per_sm * num_sms;
}

inline int warp_grid(int64_t chunk_bound, int cap) {
    const int64_t need = (chunk_bound + (kWarpThreads / 32) - 1) / (kWarpThreads / 32);
    return static_cast<int>(max64(1, min64(need, cap)));
}

// ---------------------------------------------------------------- optimizer step

// Start of a stored row.
__device__ __forceinline__ char* row_ptr(const TableDev& td, int64_t row) {
    return static_cast<char*>(const_cast<void*>(td.data)) + row * td.dim * dtype_bytes(td.dtype);
}

// The stored bits of four consecutive columns of a row: 16 bytes (fp32) or
// 8 bytes in .x, .y (fp16 / bf16).
__device__ __forceinline__ uint4 load_cols(const char* rowp, int dtype, int col) {
    if (dtype == CB_F32) return *reinterpret_cast<const uint4*>(rowp + 4 * col);
    const uint2 x = *reinterpret_cast<const uint2*>(rowp + 2 * col);
    return make_uint4(x.x, x.y, 0u, 0u);
}

// new = E - scale * g for the four columns whose stored bits are `x`, rounded
// once from fp32 to the storage type (round to nearest even), and stored.
__device__ __forceinline__ void store_step(char* rowp, int dtype, int col, uint4 x, float4 g, float scale) {
    if (dtype == CB_F32) {
        float4 v = make_float4(__uint_as_float(x.x), __uint_as_float(x.y), __uint_as_float(x.z),
                               __uint_as_float(x.w));
        v.x = fmaf(-scale, g.x, v.x);
        v.y = fmaf(-scale, g.y, v.y);
        v.z = fmaf(-scale, g.z, v.z);
        v.w = fmaf(-scale, g.w, v.w);
        *reinterpret_cast<float4*>(rowp + 4 * col) = v;
        return;
    }
    uint2 y;
    if (dtype == CB_F16) {
        __half2 a, b;
        memcpy(&a, &x.x, 4);
        memcpy(&b, &x.y, 4);
        const float2 fa = __half22float2(a), fb = __half22float2(b);
        a = __floats2half2_rn(fmaf(-scale, g.x, fa.x), fmaf(-scale, g.y, fa.y));
        b = __floats2half2_rn(fmaf(-scale, g.z, fb.x), fmaf(-scale, g.w, fb.y));
        memcpy(&y.x, &a, 4);
        memcpy(&y.y, &b, 4);
    } else {
        const float f0 = __uint_as_float(x.x << 16), f1 = __uint_as_float(x.x & 0xffff0000u);
        const float f2 = __uint_as_float(x.y << 16), f3 = __uint_as_float(x.y & 0xffff0000u);
        const __nv_bfloat162 a = __floats2bfloat162_rn(fmaf(-scale, g.x, f0), fmaf(-scale, g.y, f1));
        const __nv_bfloat162 b = __floats2bfloat162_rn(fmaf(-scale, g.z, f2), fmaf(-scale, g.w, f3));
        memcpy(&y.x, &a, 4);
        memcpy(&y.y, &b, 4);
    }
    *reinterpret_cast<uint2*>(rowp + 2 * col) = y;
}

__device__ __forceinline__ void step_cols(const TableDev& td, int64_t row, int col, float4 g, float scale) {
    char* p = row_ptr(td, row);
    store_step(p, td.dtype, col, load_cols(p, td.dtype, col), g, scale);
}

// This lane's share of sum g^2 over four columns, in one fixed order of
// roundings (an explicit product and three fused multiply-adds): written as a
// plain sum of products, the compiler may fuse either product of a pair, and
// may choose differently in the fused and the two-pass step, which must give
// the same Adagrad state bit for bit.
__device__ __forceinline__ float sq4(float4 g) {
    return fmaf(g.w, g.w, fmaf(g.z, g.z, fmaf(g.y, g.y, __fmul_rn(g.x, g.x))));
}

// The Adagrad scale from the summed squares and the row's previous state `m0`
// (meaningful in lane 0); lane 0 stores the new state.
__device__ __forceinline__ float adagrad_scale(const BwdOut& O, float* st, int dim, float sq, float m0) {
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) sq += __shfl_xor_sync(kFull, sq, off);
    float m = 0.f;
    if ((threadIdx.x & 31) == 0) {
        m = m0 + sq / static_cast<float>(dim);
        *st = m;
    }
    m = __shfl_sync(kFull, m, 0);
    return O.lr / (sqrtf(m) + O.eps);
}

// The step's scale for one row: lr (SGD), or lr / (sqrt(m) + eps) after
// m += mean of the squared gradient (row-wise Adagrad). `sq` is this lane's
// share of sum g^2; the whole warp calls this, lane 0 owns the state word.
__device__ __forceinline__ float step_scale(const BwdOut& O, int t, int64_t row, int dim, float sq) {
    if (O.apply != kApplyAdagrad) return O.lr;
    float* st = O.state[t] + row;
    return adagrad_scale(O, st, dim, sq, (threadIdx.x & 31) == 0 ? *st : 0.f);
}

// The fused step on one complete run's row, as the walker holds it: lane v of
// each row group owns vectors v + 32k; every group holds the same totals and
// group 0 writes. Out of line: the walker ends runs in many places, and a copy
// of the step in each of them overflowed the instruction cache (measured on
// cfg5: fused SGD step 36.8 ms inline, 21 ms out of line).
template <int N>
struct GradRow {
    float4 v[N];   // four gradient columns each
    int col[N];    // first column of each, or -1 past the row
};

template <int N>
__device__ __noinline__ void apply_row(const Problem& P, const BwdOut& O, int t, int32_t seg,
                                       const GradRow<N> g, bool group0) {
    const TableDev& td = P.tables[t];
    const int64_t row = static_cast<int64_t>(__ldg(O.uniq + seg)) - td.key_base;
    float sq = 0.f;
#pragma unroll
    for (int k = 0; k < N; ++k)
        if (group0 && g.col[k] >= 0)
            sq += sq4(g.v[k]);
    const float scale = step_scale(O, t, row, td.dim, sq);
    if (!group0) return;
#pragma unroll
    for (int k = 0; k < N; ++k)
        if (g.col[k] >= 0) step_cols(td, row, g.col[k], g.v[k], scale);
}

// ---------------------------------------------------------------- (5) reduce

// APPLY: the optimizer step is fused where a run's sum ends (compiled as its
// own kernels, so the gradient-writing reduce carries none of its code).
template <int GO, int VPL, bool PACKED, bool APPLY>
struct BwdPolicy {
    static constexpr int kDtype = GO;  // grad_out storage: fp32, or fp16 / bf16 (mixed precision)
    static constexpr int kElems = Storage<GO>::kElems;
    static constexpr bool kTwoLevel = true;  // gradients keep the fp32 bound for every grad_out type
    static constexpr int kVpl = VPL;
    // Half grad_out rows (8 values per lane, usually 2 rows per warp step) take
    // the forward's code shape: fewer rows in flight, one copy of the run-end
    // code per batch.
    static constexpr int kRows = APPLY ? CB_REDUCE_APPLY_ROWS : (GO == CB_F32 ? CB_REDUCE_ROWS : CB_REDUCE_HALF_ROWS);
    static constexpr int kUnroll = kRows / VPL > 0 ? kRows / VPL : 1;
    static constexpr bool kWeighted = PACKED;
    static constexpr bool kUnrollGroups = GO == CB_F32 ? CB_REDUCE_UNROLL_GROUPS : false;
    static constexpr bool kFastBatch = GO == CB_F32 ? CB_REDUCE_FAST_BATCH : CB_REDUCE_HALF_FAST_BATCH;
    static constexpr int kPrefetch = CB_REDUCE_PREFETCH;

    const Problem& P;  // kernel parameters: read in place, not held in registers
    const Plan& Q;
    const BwdOut& O;
    const uint4* base;  // grad_out + Doff_t, one row per bag of this table
    int64_t float_lo;   // first float of this table in grads
    uint32_t stride;    // 16-byte vectors per grad_out row
    int32_t chunk;
    int32_t bag_lo;
    int32_t seg_lo;     // first run of this table
    int32_t out_shift;  // run index - output row (runs of out-of-range lookups of
                        // earlier tables are not output)
    int32_t dim;
    int32_t table;

    __device__ __forceinline__ int64_t seg_begin(int32_t s) const { return __ldg(O.seg_start + s); }
    __device__ __forceinline__ int64_t seg_end(int32_t s) const { return __ldg(O.seg_start + s + 1); }
    struct Raw {
        uint32_t v;
    };
    __device__ __forceinline__ static Raw none() { return {0xffffffffu}; }
    __device__ __forceinline__ Raw fetch(int64_t q) const { return {load_stream(O.vals_sorted + q)}; }
    static constexpr int kStageBytes = 4;
    __device__ __forceinline__ void stage(char* dst, int64_t q) const { cp_async4(dst, O.vals_sorted + q); }
    __device__ __forceinline__ Raw staged(const char* src) const {
        return {*reinterpret_cast<const uint32_t*>(src)};
    }
    // Sorted item: the bag whose grad_out row it gathers, and w_i * s_b.
    __device__ __forceinline__ void decode(const Raw& x, uint32_t& a, float& w) const {
        int64_t bag;
        if (PACKED) {
            if (x.v >= P.n) {  // only after an aborted sort pass: skip the item
                a = kInvalid;
                w = 0.f;
                return;
            }
            const uint2 pk = __ldg(O.packed + x.v);
            bag = pk.x;
            w = __uint_as_float(pk.y);
        } else {
            bag = x.v;
            w = 1.f;
        }
        const int64_t b = bag - bag_lo;
        a = (b >= 0 && b < P.B) ? static_cast<uint32_t>(b) : kInvalid;
    }
    static constexpr bool kEmptySegments = false;
    // Row id (row_base_t + r = key - t) and float offset of a run that begins
    // in this chunk, at its output row.
    __device__ __forceinline__ void seg_meta(int32_t seg) const {
        if (APPLY) return;  // a fused step writes no gradient buffers
        O.unique_ids[seg - out_shift] = static_cast<int64_t>(__ldg(O.uniq + seg)) - table;
        O.grad_offsets[seg - out_shift] = float_lo + static_cast<int64_t>(seg - seg_lo) * dim;
    }
    __device__ __forceinline__ void put_empty(int32_t, int, bool) const {}
    __device__ __forceinline__ void emit(int32_t seg, int32_t L, bool started, bool ends,
                                         float (&tot)[VPL][kElems], int v, bool group0) const {
        if (started && (threadIdx.x & 31) == 0) seg_meta(seg);
        put(seg, L, started, ends, tot, v, group0);
    }
    // Lane v of a row group holds vectors v + 32k of the grad_out row: columns
    // [(v + 32k) * kElems, + kElems), written as fp32 gradients.
    __device__ __forceinline__ void put(int32_t seg, int32_t, bool started, bool ends,
                                        float (&tot)[VPL][kElems], int v, bool group0) const {
        const int64_t fo = float_lo + static_cast<int64_t>(seg - seg_lo) * dim;
        if (started && !ends && (threadIdx.x & 31) == 0) Q.tail_owner[chunk] = seg;
        if constexpr (APPLY) {
            if (started && ends) {
                GradRow<VPL * kElems / 4> r;
#pragma unroll
                for (int k = 0; k < VPL; ++k)
#pragma unroll
                    for (int x = 0; x < kElems / 4; ++x) {
                        const int col = (v + 32 * k) * kElems + 4 * x;
                        r.v[k * (kElems / 4) + x] = make_float4(tot[k][4 * x], tot[k][4 * x + 1],
                                                                tot[k][4 * x + 2], tot[k][4 * x + 3]);
                        r.col[k * (kElems / 4) + x] = col < dim ? col : -1;
                    }
                apply_row<VPL * kElems / 4>(P, O, table, seg, r, group0);
                return;
            }
        }
        if (!group0) return;
        float* dst;
        if (started && ends) dst = O.grads + fo;
        else dst = (started ? Q.carry_tail : Q.carry_head) + static_cast<int64_t>(chunk) * P.dmax;
#pragma unroll
        for (int k = 0; k < VPL; ++k) {
            const int vec = v + 32 * k;
            if (vec * kElems < dim) {
                float4* d4 = reinterpret_cast<float4*>(dst + vec * kElems);
#pragma unroll
                for (int x = 0; x < kElems / 4; ++x)
                    store_stream(d4 + x, make_float4(tot[k][4 * x], tot[k][4 * x + 1], tot[k][4 * x + 2],
                                                     tot[k][4 * x + 3]));
            }
        }
    }
};

// Resident blocks per SM the reduce is compiled for: half-precision grad_out
// slices with one vector per lane, no coefficient and no optimizer step fit 5
// blocks' registers (48) without spilling, and more resident warps raise the
// rate of the L2-served gathers; the optimizer-step form runs 5 blocks with
// 2 rows in flight (CB_REDUCE_APPLY_ROWS); fp32 slices (8 rows in flight per
// lane, whose uniform-index gathers come from DRAM and want the bytes in
// flight) and the other forms keep CB_REDUCE_MIN_BLOCKS.
#ifndef CB_REDUCE_HALF_MIN_BLOCKS
#define CB_REDUCE_HALF_MIN_BLOCKS 5
#endif
#ifndef CB_REDUCE_APPLY_MIN_BLOCKS
#define CB_REDUCE_APPLY_MIN_BLOCKS 5  // the reduce with the optimizer step fused
#endif
template <int GO, int VPL, bool PACKED, int GC, bool APPLY>
constexpr int reduce_min_blocks() {
    if (APPLY) return CB_REDUCE_APPLY_MIN_BLOCKS;
    return GO != CB_F32 && VPL == 1 && GC > 0 && GC != 4 && !PACKED ? CB_REDUCE_HALF_MIN_BLOCKS
                                                                    : CB_REDUCE_MIN_BLOCKS;
}

template <int GO, int VPL, bool PACKED, int GC, bool APPLY>
__global__ void __launch_bounds__(kWarpThreads, reduce_min_blocks<GO, VPL, PACKED, GC, APPLY>())
    bwd_reduce_kernel(const __grid_constant__ Problem P, const __grid_constant__ Plan Q,
                      const __grid_constant__ BwdOut O, const void* grad_out, int cls) {
    if (*O.cap_fail) return;
    const int lane = threadIdx.x & 31;
    const int64_t cb = Q.class_chunk_base[cls];
    const int64_t ce = min64(Q.class_chunk_base[cls + 1], Q.max_chunks);
    for (int64_t j = first_chunk(Q, cls, cb, lane); j < ce;) {
        const int64_t nxt = fetch_next_chunk(Q, cls, cb, lane);
        const Chunk ch = Q.chunks[j];
        const int t = ch.table;
        const TableDev& td = P.tables[t];
        BwdPolicy<GO, VPL, PACKED, APPLY> pol{P, Q, O};
        constexpr int eb = GO == CB_F32 ? 4 : 2;
        pol.base = reinterpret_cast<const uint4*>(static_cast<const char*>(grad_out) +
                                                  static_cast<int64_t>(td.doff) * eb);
        pol.float_lo = O.float_base[t];
        pol.stride = static_cast<uint32_t>(P.sum_d * eb / 16);
        pol.chunk = static_cast<int32_t>(j);
        pol.bag_lo = t * P.B;
        pol.seg_lo = static_cast<int32_t>(O.table_first[t]);
        pol.out_shift = static_cast<int32_t>(O.table_first[t] - O.out_first[t]);
        pol.dim = td.dim;
        pol.table = t;
        ChunkCtx c;
        c.k0 = ch.k0;
        c.len = static_cast<int32_t>(ch.len & 0x7fffffffu);
        c.first = static_cast<int32_t>(max64(ch.first, O.table_first[t]));
        // The run of out-of-range lookups (the table's spare key, last) is
        // walked but never output: its items read the zero row.
        c.seg_hi = static_cast<int32_t>(O.live_end[t]);
        c.lanes = td.grad_lanes;
        c.groups = td.grad_groups;
        c.row_vecs = td.grad_vecs;
        c.last = false;
        if (lane == 0) Q.tail_owner[j] = -1;
        if constexpr (GC > 0 && VPL == 1 && CB_ROW_WALKER) {
            __shared__ EndSlot slots[kWarpThreads / 32][32];
#if defined(CB_REDUCE_STAGE) && CB_REDUCE_STAGE > 0
            __shared__ __align__(16) char stage[kWarpThreads / 32][(CB_REDUCE_STAGE + 1) * 32 * 4];
            walk_rows<BwdPolicy<GO, VPL, PACKED, APPLY>, GC, 0, CB_REDUCE_STAGE>(
                pol, c, P.zero_row, lane, slots[threadIdx.x >> 5], nullptr, stage[threadIdx.x >> 5]);
#else
            walk_rows<BwdPolicy<GO, VPL, PACKED, APPLY>, GC>(pol, c, P.zero_row, lane, slots[threadIdx.x >> 5]);
#endif
        } else {
            walk_chunk<BwdPolicy<GO, VPL, PACKED, APPLY>, GC>(pol, c, P.zero_row, lane);
        }
        j = __shfl_sync(kFull, nxt, 0);
    }
}

template <int GO, int VPL, bool PACKED, int GC, bool APPLY>
static void launch_reduce_one(const Problem& P, const Plan& Q, const BwdOut& O, const void* go,
                              int cls, int64_t chunk_bound, int num_sms, cudaStream_t s) {
    static int cap = occupancy_grid(bwd_reduce_kernel<GO, VPL, PACKED, GC, APPLY>, kWarpThreads, num_sms);
    bwd_reduce_kernel<GO, VPL, PACKED, GC, APPLY><<<warp_grid(chunk_bound, cap), kWarpThreads, 0, s>>>(
        P, Q, O, go, cls);
}

template <int GO, bool APPLY>
void launch_bwd_reduce_t(const Problem& P, const Plan& Q, const BwdOut& O, const void* grad_out,
                         int cls, int vpl, int gc, bool packed, int64_t chunk_bound, int num_sms,
                         cudaStream_t s) {
#define CB_CASE(V, G, PK)                                                                \
    if (vpl == V && gc == G && packed == PK) {                                            \
        launch_reduce_one<GO, V, PK, G, APPLY>(P, Q, O, grad_out, cls, chunk_bound, num_sms, s); \
        return;                                                                          \
    }
    CB_CASE(1, 1, false) CB_CASE(1, 2, false) CB_CASE(1, 4, false) CB_CASE(1, 8, false)
    CB_CASE(1, 0, false) CB_CASE(2, 1, false) CB_CASE(4, 1, false)
    CB_CASE(1, 1, true) CB_CASE(1, 2, true) CB_CASE(1, 4, true) CB_CASE(1, 8, true)
    CB_CASE(1, 0, true) CB_CASE(2, 1, true) CB_CASE(4, 1, true)
#undef CB_CASE
}

}  // namespace cbtbe
