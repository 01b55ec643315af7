// tbe_forward.cuh -- forward gather-pool kernel template of the pooled
// embedding bag (sparse_arch lookups, Sec. IV.A.2; jagged categorical features,
// Abstract):
//   out[b, Doff_t + j] = s_b * sum_{i in bag(t, b)} w_i * E_t[indices[i], j]
//
// One warp per chunk of lookup positions. A stored row is spread over V lanes
// (16 bytes per lane per vector, V = row bytes / 16 up to 32), and a warp step
// gathers G = 32 / V rows of the chunk at once, each lane keeping several
// 16-byte loads in flight. Rows widen to fp32 in registers; the G per-row
// partial sums of a bag meet through warp shuffles when the bag is emitted.
// Instantiated per storage type in tbe_forward_{f32,f16,bf16}.cu.
#pragma once

#include "tbe_internal.cuh"
#include "tbe_launch.h"

namespace cbtbe {

template <int DT, int VPL, bool WEIGHTED>
struct FwdPolicy {
    static constexpr int kDtype = DT;
    static constexpr int kElems = Storage<DT>::kElems;
    static constexpr int kVpl = VPL;
    static constexpr int kUnroll = CB_WALK_ROWS / VPL > 0 ? CB_WALK_ROWS / VPL : 1;
    static constexpr bool kWeighted = WEIGHTED;
    static constexpr bool kTwoLevel = DT == CB_F32;  // half rows: one fp32 level (registers)
    static constexpr bool kUnrollGroups = CB_WALK_UNROLL_GROUPS;
    static constexpr bool kFastBatch = CB_WALK_FAST_BATCH;
    static constexpr int kPrefetch = CB_WALK_PREFETCH;

    const Problem& P;  // kernel parameters: read in place, not held in registers
    const Plan& Q;
    void* out;         // [B, sum D] of P.out_dtype
    const uint4* base;  // the table
    int64_t rows;
    uint32_t stride;    // 16-byte vectors per row
    int32_t row_vecs;
    int32_t chunk;
    int32_t bag_lo;
    int32_t doff;

    __device__ __forceinline__ int64_t seg_begin(int32_t s) const { return load_index(P.offsets, s, P.is32); }
    __device__ __forceinline__ int64_t seg_end(int32_t s) const { return load_index(P.offsets, s + 1, P.is32); }
    struct Raw {
        int64_t r;
        float w;
    };
    __device__ __forceinline__ static Raw none() { return {-1, 0.f}; }
    __device__ __forceinline__ Raw fetch(int64_t q) const {
        return {load_index(P.indices, q, P.is32), WEIGHTED ? __ldg(P.weights + q) : 1.f};
    }
    // The same payload staged in shared memory (index in the first 8 bytes, the
    // weight after it).
    static constexpr int kStageBytes = WEIGHTED ? 16 : 8;
    __device__ __forceinline__ void stage(char* dst, int64_t q) const {
        if (P.is32) cp_async4(dst, static_cast<const int*>(P.indices) + q);
        else cp_async8(dst, static_cast<const long long*>(P.indices) + q);
        if (WEIGHTED) cp_async4(dst + 8, P.weights + q);
    }
    __device__ __forceinline__ Raw staged(const char* src) const {
        const int64_t r = P.is32 ? static_cast<int64_t>(*reinterpret_cast<const int*>(src))
                                 : static_cast<int64_t>(*reinterpret_cast<const long long*>(src));
        return {r, WEIGHTED ? *reinterpret_cast<const float*>(src + 8) : 1.f};
    }
    // Row id of a lookup, checked once here; an out-of-range id contributes nothing.
    __device__ __forceinline__ void decode(const Raw& x, uint32_t& a, float& w) const {
        w = x.w;
        if (x.r < 0 || x.r >= rows) {
            set_error(P.error, CB_ERR_INDEX_OOB);
            a = kInvalid;
        } else {
            a = static_cast<uint32_t>(x.r);
        }
    }
    static constexpr bool kEmptySegments = true;
    __device__ __forceinline__ void seg_meta(int32_t) const {}
    __device__ __forceinline__ void put(int32_t bag, int32_t L, bool started, bool ends,
                                        float (&tot)[VPL][kElems], int v, bool group0) const {
        emit(bag, L, started, ends, tot, v, group0);
    }
    // An empty bag pools to zeros (one vector per lane).
    __device__ __forceinline__ void put_empty(int32_t bag, int v, bool group0) const {
        if (!group0) return;
        const int64_t col = static_cast<int64_t>(bag - bag_lo) * P.sum_d + doff + v * kElems;
#pragma unroll
        for (int x = 0; x < kElems / 4; ++x) store_out4(out, col + 4 * x, 0.f, 0.f, 0.f, 0.f, P.out_dtype);
    }
    __device__ __forceinline__ void emit(int32_t bag, int32_t L, bool started, bool ends,
                                         float (&tot)[VPL][kElems], int v, bool group0) const {
        if (started && !ends && (threadIdx.x & 31) == 0) Q.tail_owner[chunk] = bag;
        if (!group0) return;
        if (started && ends) {
            // A complete bag: the pooled row, in the output's type.
            if (P.mean && L > 0) {
                const float scale = static_cast<float>(L);
#pragma unroll
                for (int k = 0; k < VPL; ++k)
#pragma unroll
                    for (int x = 0; x < kElems; ++x) tot[k][x] = tot[k][x] / scale;
            }
            const int64_t col0 = static_cast<int64_t>(bag - bag_lo) * P.sum_d + doff;
#pragma unroll
            for (int k = 0; k < VPL; ++k) {
                const int vec = v + 32 * k;
                if (vec >= row_vecs) continue;
#pragma unroll
                for (int x = 0; x < kElems / 4; ++x)
                    store_out4(out, col0 + vec * kElems + 4 * x, tot[k][4 * x], tot[k][4 * x + 1],
                               tot[k][4 * x + 2], tot[k][4 * x + 3], P.out_dtype);
            }
            return;
        }
        // A piece of a bag split across chunks: fp32, for the fix-up.
        float* dst = (started ? Q.carry_tail : Q.carry_head) + static_cast<int64_t>(chunk) * P.dmax;
#pragma unroll
        for (int k = 0; k < VPL; ++k) {
            const int vec = v + 32 * k;
            if (vec >= row_vecs) continue;
            float4* d4 = reinterpret_cast<float4*>(dst + vec * kElems);
#pragma unroll
            for (int x = 0; x < kElems / 4; ++x)
                d4[x] = make_float4(tot[k][4 * x], tot[k][4 * x + 1], tot[k][4 * x + 2], tot[k][4 * x + 3]);
        }
    }
};

// Groups of row loads kept in flight per warp through shared memory by the
// row walker (0: loads into registers).
#ifndef CB_GATHER_ASYNC
#define CB_GATHER_ASYNC 0
#endif
constexpr int kGatherAsync = CB_GATHER_ASYNC;
// Batches of lookup payloads (indices, weights) staged ahead in shared memory
// by cp.async (0: loaded into registers one batch ahead).
#ifndef CB_INDEX_STAGE
#define CB_INDEX_STAGE 0
#endif
constexpr int kIndexStage = CB_INDEX_STAGE;

// 16-byte slots per lane of a warp's ring: (groups in flight + 1) load groups.
template <class Pol, int GC>
__host__ __device__ constexpr int gather_ring_slots() {
    constexpr int steps = GC > 0 ? 32 / GC : 1;
    constexpr int ug = Pol::kUnroll < steps ? Pol::kUnroll : steps;
    constexpr int groups = steps / ug;  // load groups per batch of 32 items
    constexpr int depth = kGatherAsync < groups ? kGatherAsync : groups;
    return kGatherAsync > 0 ? (depth + 1) * ug : 0;
}

// Resident blocks per SM the gather is compiled for. The row walker with one
// vector per lane and no weights fits 5 blocks' registers (48) without
// spilling, and the gather's rate out of L2 grows with the warps resident
// (cfg5: 4.07 -> 3.72 ms from 4 to 5 blocks); the other layouts spill at 48
// registers and keep 4.
#ifndef CB_WALK_MIN_BLOCKS_ROW
#define CB_WALK_MIN_BLOCKS_ROW 5
#endif
#ifndef CB_WALK_ROW_WEIGHTED
#define CB_WALK_ROW_WEIGHTED 0  // 1: weighted row layouts take CB_WALK_MIN_BLOCKS_ROW too
#endif
template <int VPL, bool WEIGHTED, int GC>
constexpr int gather_min_blocks() {
    return VPL == 1 && GC > 0 && GC != 4 && (!WEIGHTED || CB_WALK_ROW_WEIGHTED) ? CB_WALK_MIN_BLOCKS_ROW
                                                                                : CB_WALK_MIN_BLOCKS;
}

template <int DT, int VPL, bool WEIGHTED, int GC>
__global__ void __launch_bounds__(kWarpThreads, gather_min_blocks<VPL, WEIGHTED, GC>())
    fwd_gather_kernel(const __grid_constant__ Problem P, const __grid_constant__ Plan Q, void* out,
                      int cls) {
    const int lane = threadIdx.x & 31;
    const int64_t cb = Q.class_chunk_base[cls];
    const int64_t ce = min64(Q.class_chunk_base[cls + 1], Q.max_chunks);
    for (int64_t j = first_chunk(Q, cls, cb, lane); j < ce;) {
        const int64_t nxt = fetch_next_chunk(Q, cls, cb, lane);
        const Chunk ch = Q.chunks[j];
        const TableDev& td = P.tables[ch.table];
        FwdPolicy<DT, VPL, WEIGHTED> pol{P, Q, out};
        pol.base = static_cast<const uint4*>(td.data);
        pol.rows = td.rows;
        pol.stride = static_cast<uint32_t>(td.row_vecs);
        pol.row_vecs = td.row_vecs;
        pol.chunk = static_cast<int32_t>(j);
        pol.bag_lo = ch.table * P.B;
        pol.doff = td.doff;
        ChunkCtx c;
        c.k0 = ch.k0;
        c.len = static_cast<int32_t>(ch.len & 0x7fffffffu);
        c.first = static_cast<int32_t>(ch.first);
        c.seg_hi = pol.bag_lo + P.B;
        c.lanes = td.lanes;
        c.groups = td.groups;
        c.row_vecs = td.row_vecs;
        c.last = (ch.len >> 31) != 0;
        if (lane == 0) Q.tail_owner[j] = -1;
        if constexpr (GC > 0 && VPL == 1 && CB_ROW_WALKER) {
            __shared__ EndSlot slots[kWarpThreads / 32][32];
            if constexpr (kGatherAsync > 0) {
                extern __shared__ __align__(16) uint4 ring[];
                constexpr int kSlots = gather_ring_slots<FwdPolicy<DT, VPL, WEIGHTED>, GC>();
                walk_rows<FwdPolicy<DT, VPL, WEIGHTED>, GC, kGatherAsync>(
                    pol, c, P.zero_row, lane, slots[threadIdx.x >> 5], ring + (threadIdx.x >> 5) * kSlots * 32);
            } else if constexpr (kIndexStage > 0) {
                using Pol = FwdPolicy<DT, VPL, WEIGHTED>;
                __shared__ __align__(16) char stage[kWarpThreads / 32][(kIndexStage + 1) * 32 * Pol::kStageBytes];
                walk_rows<Pol, GC, 0, kIndexStage>(pol, c, P.zero_row, lane, slots[threadIdx.x >> 5], nullptr,
                                                  stage[threadIdx.x >> 5]);
            } else {
                walk_rows<FwdPolicy<DT, VPL, WEIGHTED>, GC>(pol, c, P.zero_row, lane, slots[threadIdx.x >> 5]);
            }
        } else {
            walk_chunk<FwdPolicy<DT, VPL, WEIGHTED>, GC>(pol, c, P.zero_row, lane);
        }
        j = __shfl_sync(kFull, nxt, 0);
    }
}

// Dynamic shared memory of the gather: the warps' rings of staged row loads.
template <int DT, int VPL, bool W, int GC>
static size_t gather_smem() {
    if constexpr (GC > 0 && VPL == 1 && CB_ROW_WALKER)
        return sizeof(uint4) * 32 * (kWarpThreads / 32) * gather_ring_slots<FwdPolicy<DT, VPL, W>, GC>();
    return 0;
}

template <int DT, int VPL, bool W, int GC>
static int gather_grid(int num_sms) {
    static int per_sm = -1;
    if (per_sm < 0) {
        const size_t smem = gather_smem<DT, VPL, W, GC>();
        if (smem > 0)
            cudaFuncSetAttribute(fwd_gather_kernel<DT, VPL, W, GC>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(smem));
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fwd_gather_kernel<DT, VPL, W, GC>,
                                                          kWarpThreads, smem) != cudaSuccess ||
            per_sm < 1)
            per_sm = 1;
    }
    return per_sm * num_sms;
}

template <int DT, int VPL, int GC>
static void launch_gather_layout(const Problem& P, const Plan& Q, void* out, int cls,
                                 int64_t chunk_bound, int num_sms, cudaStream_t s) {
    const int64_t need = (chunk_bound + (kWarpThreads / 32) - 1) / (kWarpThreads / 32);
    if (P.weights) {
        const int grid = static_cast<int>(min64(need, gather_grid<DT, VPL, true, GC>(num_sms)));
        fwd_gather_kernel<DT, VPL, true, GC><<<max(grid, 1), kWarpThreads, gather_smem<DT, VPL, true, GC>(), s>>>(
            P, Q, out, cls);
    } else {
        const int grid = static_cast<int>(min64(need, gather_grid<DT, VPL, false, GC>(num_sms)));
        fwd_gather_kernel<DT, VPL, false, GC><<<max(grid, 1), kWarpThreads, gather_smem<DT, VPL, false, GC>(), s>>>(
            P, Q, out, cls);
    }
}

// Row layouts compiled for: (vectors per lane, rows per step) =
// (1, 1|2|4|8), (2, 1), (4, 1), and (1, run-time) for odd row sizes.
template <int DT>
void launch_gather_dtype(const Problem& P, const Plan& Q, void* out, int cls, int vpl, int gc,
                         int64_t chunk_bound, int num_sms, cudaStream_t s) {
#define CB_CASE(V, G)                                                                \
    if (vpl == V && gc == G) {                                                        \
        launch_gather_layout<DT, V, G>(P, Q, out, cls, chunk_bound, num_sms, s);      \
        return;                                                                      \
    }
    CB_CASE(1, 1) CB_CASE(1, 2) CB_CASE(1, 4) CB_CASE(1, 8) CB_CASE(1, 0)
    CB_CASE(2, 1) CB_CASE(4, 1)
#undef CB_CASE
}

}  // namespace cbtbe
