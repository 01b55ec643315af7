// tbe_internal.cuh -- device-side structures and the segmented gather-reduce
// walker shared by the forward gather-pool and the backward segmented reduce.
//
// Both hot loops have the same shape: a run of items in position order, grouped
// into consecutive segments (forward: the bags of a table, delimited by the
// jagged offsets; backward: runs of equal sorted row ids), where each item names
// a row to gather and a scalar coefficient, and each segment's output is the
// coefficient-weighted sum of its rows. The pooled bag of the paper's sparse_arch
// (Sec. IV.A.2) and its de-duplicated adjoint are both this shape.
//
// Work is cut into fixed-size chunks of item positions, so every warp does the
// same amount of gathering whatever the bag-length distribution (heavy tails,
// empty bags, one-hot bags). A segment that straddles chunk boundaries is summed
// piecewise; its pieces are combined afterwards in chunk order, in fp64, by a
// fix-up pass, so results are deterministic.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_fp16.h>
#include <cuda_bf16.h>
#include <type_traits>

#include "cb_tbe.h"

namespace cbtbe {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kWarpThreads = 256;  // block size of the warp-per-chunk kernels
#ifndef CB_WALK_MIN_BLOCKS
#define CB_WALK_MIN_BLOCKS 4  // resident blocks per SM the walker kernels are compiled for
#endif
#ifndef CB_WALK_ROWS
#define CB_WALK_ROWS 4  // 16-byte rows in flight per lane in the walker (with one vector per lane)
#endif
// Load groups ahead whose rows are prefetched into L1 (0: none), per kernel
// (measured on cfg5 / cfg5u): the Zipf gather slows down by 2.4x with one
// group ahead (its hot rows already live in L1), the reduce gains ~1 %.
#ifndef CB_WALK_PREFETCH
#define CB_WALK_PREFETCH 0
#endif
#ifndef CB_REDUCE_PREFETCH
#define CB_REDUCE_PREFETCH 1
#endif
#ifndef CB_REDUCE_MIN_BLOCKS
#define CB_REDUCE_MIN_BLOCKS 3  // the backward reduce's own targets (from the same sweep)
#endif
#ifndef CB_REDUCE_ROWS
#define CB_REDUCE_ROWS 8
#endif
// Row-walker code shape, per kernel (measured on cfg5): the forward keeps one
// copy of the segment-end code per batch (unrolling it over the load groups
// overflowed the instruction cache and doubled the gather time) and, since
// warps take chunks from a counter, no separate unrolled path for batches with
// no segment end either (gather 4.74 -> 4.49 ms without it); the fp32 backward
// reduce also keeps one copy of its run-end code per batch but unrolls the
// batches with no run end (reduce 5.40 -> 5.19 ms on cfg5; 18.45 -> 18.59 ms on
// uniform indices, where nearly every batch has run ends).
#ifndef CB_WALK_UNROLL_GROUPS
#define CB_WALK_UNROLL_GROUPS 0
#endif
#ifndef CB_WALK_FAST_BATCH
#define CB_WALK_FAST_BATCH 0
#endif
#ifndef CB_REDUCE_UNROLL_GROUPS
#define CB_REDUCE_UNROLL_GROUPS 0
#endif
#ifndef CB_REDUCE_FAST_BATCH
#define CB_REDUCE_FAST_BATCH 1
#endif
#ifndef CB_ROW_WALKER
#define CB_ROW_WALKER 1  // 0: every layout takes the general walker (walk_chunk)
#endif
constexpr int64_t kNoSeg = INT64_MAX;

// Per-table facts the kernels need, built once at create time.
struct TableDev {
    const void* data;   // row-major [rows, dim] of dtype
    int64_t rows;
    int64_t row_base;   // rows of all tables before this one (global row id base)
    // Backward sort key of row r: key_base + r, with key_base = row_base + t.
    // Each table owns rows + 1 keys; key_base + rows marks a lookup whose index
    // is out of range, which sorts after the table's rows into a run of its own
    // that the reduce drops.
    int64_t key_base;
    int32_t dim;
    int32_t doff;       // column offset of this table in the [B, sum dims] output
    int32_t dtype;      // cb_dtype
    int32_t row_vecs;   // 16-byte vectors per stored row
    int32_t lanes;      // lanes per stored row in the gather (V)
    int32_t groups;     // stored rows per warp step (G, V * G <= 32)
    int32_t grad_vecs;  // 16-byte vectors per fp32 gradient row (dim / 4)
    int32_t grad_lanes;
    int32_t grad_groups;
    int32_t fwd_class;
    int32_t bwd_class;
    int32_t pad;
};

// A run of at most chunk_len item positions of one table.
struct Chunk {
    int64_t k0;     // first item position
    int64_t first;  // first segment touching k0 (bag id, or unique-row index)
    int32_t table;
    uint32_t len;   // bit 31: last chunk of its table; bits 0..30: item count
};

struct Problem {
    const TableDev* tables;
    const uint4* zero_row;  // 2 KB of zeros: the row an invalid or padding item reads
    const void* indices;
    const void* offsets;
    const float* weights;
    int* error;
    int64_t n;
    int32_t T;
    int32_t B;
    int32_t sum_d;
    int32_t is32;
    int32_t mean;
    int32_t dmax;  // largest dim (row stride of the carry buffers)
    int32_t out_dtype;  // cb_dtype of the pooled output and of grad_out
};

struct Plan {
    int32_t chunk_len;
    int32_t snap_cap;                  // segments up to this long are never split (0: no snapping)
    int32_t num_classes;
    const int32_t* class_tables;       // [T] table ids grouped by kernel class
    const int32_t* class_table_start;  // [num_classes + 1]
    int64_t* table_pos;                // [T + 1] first item position of each table
    int64_t* ord_chunk_base;           // [T + 1] first chunk of class_tables[i]
    int64_t* class_chunk_base;         // [num_classes + 1]
    Chunk* chunks;                     // [max_chunks]
    int64_t max_chunks;
    float* carry_head;                 // [max_chunks, dmax] piece of a segment begun earlier
    float* carry_tail;                 // [max_chunks, dmax] piece of a segment begun here
    int64_t* tail_owner;               // [max_chunks] segment whose tail piece is here, or -1
    uint32_t* chunk_next;              // [num_classes + 1] next chunk to hand out per class, and
                                       // over all classes (zeroed by the plan)
};


__host__ __device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }
__host__ __device__ __forceinline__ int64_t max64(int64_t a, int64_t b) { return a > b ? a : b; }

__device__ __forceinline__ void set_error(int* err, int code) { atomicCAS(err, 0, code); }

__device__ __forceinline__ int64_t load_index(const void* p, int64_t i, int is32) {
    return is32 ? static_cast<int64_t>(__ldg(static_cast<const int*>(p) + i))
                : static_cast<int64_t>(__ldg(static_cast<const long long*>(p) + i));
}

__device__ __forceinline__ int64_t warp_id_global() {
    return (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
}
__device__ __forceinline__ int64_t warps_in_grid() {
    return (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
}

// The walkers' chunk order: a warp takes the next chunk of its class from a
// counter (lane 0 fetches the one after while the warp walks the current one),
// so chunks start in order and cheap chunks do not leave warps idle.
__device__ __forceinline__ int64_t first_chunk(const Plan& Q, int cls, int64_t cb, int lane) {
    const int64_t j = lane == 0 ? cb + atomicAdd(Q.chunk_next + cls, 1u) : 0;
    return __shfl_sync(kFull, j, 0);
}
__device__ __forceinline__ int64_t fetch_next_chunk(const Plan& Q, int cls, int64_t cb, int lane) {
    return lane == 0 ? cb + atomicAdd(Q.chunk_next + cls, 1u) : 0;
}

// ---------------------------------------------------------------- bags of positions

// The bag of each of 32 consecutive lookup positions of one table. A window of
// 32 bag ends slides forward (lane i holds the end of bag win + i); ends never
// decrease (valid offsets), so the number of the window's bags that end at or
// before a position is a bisection. Each lane gets its bag and the bag's
// [start, end) positions.
struct BagWindow {
    int64_t win;        // first bag of the window
    int64_t win_start;  // start position of bag win
    int64_t my_end;     // end position of bag win + lane (kNoSeg past the table)
    int64_t bag_hi;     // one past the table's last bag
};

__device__ __forceinline__ BagWindow bag_window(const Problem& P, int64_t first, int64_t bag_hi,
                                                int lane) {
    BagWindow W;
    W.win = first;
    W.bag_hi = bag_hi;
    W.win_start = first < bag_hi ? load_index(P.offsets, first, P.is32) : kNoSeg;
    W.my_end = (first + lane < bag_hi) ? load_index(P.offsets, first + lane + 1, P.is32) : kNoSeg;
    return W;
}

// Every lane of the warp calls this with its position q (valid: q is a lookup
// of the table); bag = -1 for invalid lanes.
__device__ __forceinline__ void find_bag(const Problem& P, BagWindow& W, int64_t q, bool valid, int lane,
                                         int64_t& bag, int64_t& s, int64_t& e) {
    bag = -1;
    s = e = 0;
    while (true) {
        int cnt = 0;
#pragma unroll
        for (int b = 16; b >= 1; b >>= 1)
            if (__shfl_sync(kFull, W.my_end, cnt + b - 1) <= q) cnt += b;
        if (__shfl_sync(kFull, W.my_end, 31) <= q) cnt = 32;
        const int64_t e_sel = __shfl_sync(kFull, W.my_end, cnt < 32 ? cnt : 31);
        const int64_t s_sel = __shfl_sync(kFull, W.my_end, cnt > 0 ? cnt - 1 : 0);
        if (valid && bag < 0 && cnt < 32) {
            bag = W.win + cnt;
            e = e_sel;
            s = cnt > 0 ? s_sel : W.win_start;
        }
        if (!__any_sync(kFull, valid && bag < 0)) break;
        W.win_start = __shfl_sync(kFull, W.my_end, 31);
        W.win += 32;
        W.my_end = (W.win + lane < W.bag_hi) ? load_index(P.offsets, W.win + lane + 1, P.is32) : kNoSeg;
    }
}

// ---------------------------------------------------------------- storage types

template <int DT> struct Storage;
template <> struct Storage<CB_F32> { static constexpr int kElems = 4; };
template <> struct Storage<CB_F16> { static constexpr int kElems = 8; };
template <> struct Storage<CB_BF16> { static constexpr int kElems = 8; };

template <int DT>
__device__ __forceinline__ void unpack(const uint4& r, float (&f)[Storage<DT>::kElems]);

template <>
__device__ __forceinline__ void unpack<CB_F32>(const uint4& r, float (&f)[4]) {
    f[0] = __uint_as_float(r.x);
    f[1] = __uint_as_float(r.y);
    f[2] = __uint_as_float(r.z);
    f[3] = __uint_as_float(r.w);
}

template <>
__device__ __forceinline__ void unpack<CB_F16>(const uint4& r, float (&f)[8]) {
    const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        __half2 h;
        memcpy(&h, &w[i], 4);
        const float2 p = __half22float2(h);
        f[2 * i] = p.x;
        f[2 * i + 1] = p.y;
    }
}

// bfloat16 is the upper half of a binary32 word, so widening is a shift.
template <>
__device__ __forceinline__ void unpack<CB_BF16>(const uint4& r, float (&f)[8]) {
    const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        f[2 * i] = __uint_as_float(w[i] << 16);
        f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
}

// ---------------------------------------------------------------- output rows

// Cache hints for data touched once per call (CB_STREAM_HINTS): outputs
// stored with evict-first (st.global.cs), so that they leave L2 before the
// rows the walkers gather again, and one-pass payload streams loaded with it.
#ifndef CB_STREAM_HINTS
#define CB_STREAM_HINTS 1
#endif
__device__ __forceinline__ void store_stream(float4* p, float4 v) {
    if (CB_STREAM_HINTS) __stcs(p, v);
    else *p = v;
}
__device__ __forceinline__ void store_stream(uint2* p, uint2 v) {
    if (CB_STREAM_HINTS) __stcs(p, v);
    else *p = v;
}
__device__ __forceinline__ uint32_t load_stream(const uint32_t* p) { return CB_STREAM_HINTS ? __ldcs(p) : __ldg(p); }

// Four consecutive columns of an output row, stored as fp32 or rounded to
// fp16 / bf16 (round to nearest even).
__device__ __forceinline__ void store_out4(void* row, int64_t col, float a, float b, float c, float d,
                                           int dtype) {
    if (dtype == CB_F32) {
        store_stream(reinterpret_cast<float4*>(static_cast<float*>(row) + col), make_float4(a, b, c, d));
        return;
    }
    uint2 w;
    if (dtype == CB_F16) {
        const __half2 lo = __floats2half2_rn(a, b), hi = __floats2half2_rn(c, d);
        memcpy(&w.x, &lo, 4);
        memcpy(&w.y, &hi, 4);
    } else {
        const __nv_bfloat162 lo = __floats2bfloat162_rn(a, b), hi = __floats2bfloat162_rn(c, d);
        memcpy(&w.x, &lo, 4);
        memcpy(&w.y, &hi, 4);
    }
    store_stream(reinterpret_cast<uint2*>(static_cast<uint16_t*>(row) + col), w);
}

__host__ __device__ __forceinline__ int dtype_bytes(int dtype) { return dtype == CB_F32 ? 4 : 2; }

// ---------------------------------------------------------------- accumulation

// acc += w * row (WEIGHTED) or acc += row. Half-precision rows use the
// mixed-precision add of sm_100+ (f16/bf16 operand widened exactly, fp32 sum),
// which is the same arithmetic as widening first and then adding.
// (Measured on cfg5: widening fp16 pairs first and adding in fp32 took 29 %
// more instructions and 11 % more time; widening them and adding with one
// packed fp32x2 add, 16 % more instructions and 12 % more time.)
template <int DT, bool WEIGHTED>
__device__ __forceinline__ void accumulate(float (&a)[Storage<DT>::kElems], const uint4& x, float w) {
    const uint32_t word[4] = {x.x, x.y, x.z, x.w};
    if constexpr (DT == CB_F32) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float f = __uint_as_float(word[i]);
            a[i] = WEIGHTED ? fmaf(w, f, a[i]) : a[i] + f;
        }
    } else if constexpr (WEIGHTED) {
        float f[8];
        unpack<DT>(x, f);
#pragma unroll
        for (int i = 0; i < 8; ++i) a[i] = fmaf(w, f[i], a[i]);
    } else if constexpr (DT == CB_F16) {
#pragma unroll
        for (int i = 0; i < 4; ++i)
            asm("{ .reg .b16 lo, hi;\n\t mov.b32 {lo, hi}, %2;\n\t"
                " add.rn.f32.f16 %0, lo, %0;\n\t add.rn.f32.f16 %1, hi, %1; }"
                : "+f"(a[2 * i]), "+f"(a[2 * i + 1]) : "r"(word[i]));
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i)
            asm("{ .reg .b16 lo, hi;\n\t mov.b32 {lo, hi}, %2;\n\t"
                " add.rn.f32.bf16 %0, lo, %0;\n\t add.rn.f32.bf16 %1, hi, %1; }"
                : "+f"(a[2 * i]), "+f"(a[2 * i + 1]) : "r"(word[i]));
    }
}

// ---------------------------------------------------------------- the walker
//
// Pol (policy) supplies:
//   kDtype, kElems, kVpl (16-byte vectors per lane), kUnroll (rows in flight per
//   lane), kWeighted
//   int64_t seg_begin(s), seg_end(s)    positions of segment s (s < seg_hi)
//   Raw fetch(q), static Raw none()      raw payload of item q (loads only)
//   void decode(Raw, uint32_t& a, float& w)  row number within `base`
//                                            (kInvalid = skip) and coefficient
//   const uint4* base; uint32_t stride       row a starts at base + a * stride
//   void emit(seg, len, started, ends, tot, lane-in-group v, is_group0)
//                                            len = segment length when complete
// Positions inside the walker are relative to the chunk start and clamped to
// [kRelLo, kRelHi], which keeps every comparison with [0, len] exact in 32 bits.
// The segment range of the chunk is [first, seg_hi); segments that start at or
// after the chunk end belong to the next chunk, except after the last chunk of a
// table (trailing empty bags), which `last` allows.

constexpr uint32_t kInvalid = 0xffffffffu;
constexpr int32_t kRelLo = -1;
constexpr int32_t kRelHi = 1 << 30;

struct ChunkCtx {
    int64_t k0;        // absolute position of the chunk's first item
    int32_t len;       // items in the chunk
    int32_t first;     // first segment
    int32_t seg_hi;    // segments of this table end before seg_hi
    int32_t lanes;     // V
    int32_t groups;    // G
    int32_t row_vecs;  // vectors per row
    bool last;         // owns trailing segments that start at the chunk end
};

__device__ __forceinline__ int32_t rel_pos(int64_t x, int64_t k0) {
    const int64_t r = x - k0;
    return r < kRelLo ? kRelLo : (r > kRelHi ? kRelHi : static_cast<int32_t>(r));
}

// GC > 0: the row layout is known at compile time (G = GC rows per warp step,
// V = 32 / GC lanes per row); GC == 0: taken from the chunk at run time (rows
// whose vector count is not a power of two).
template <class Pol, int GC>
__device__ __forceinline__ void walk_chunk(Pol& pol, const ChunkCtx& c, const uint4* zero_row,
                                           int lane) {
    constexpr int E = Pol::kElems;
    constexpr int VPL = Pol::kVpl;
    constexpr int U = Pol::kUnroll;
    constexpr bool W = Pol::kWeighted;
    constexpr bool kExact = GC > 0 && VPL == 1;  // each lane owns one vector of one row
    const int V = GC > 0 ? 32 / GC : c.lanes;
    const int G = GC > 0 ? GC : c.groups;
    const int g = lane / V;
    const int v = lane - g * V;
    const int ustop = min(U, 32 / G);  // row groups per step
    const int step = ustop * G;        // items per step (<= 32, divides 32)
    const int32_t len = c.len;
    // Lanes past the row (non power-of-two rows) and vectors past it read zeros.
    const uint4* vzero[VPL];
    bool vlive[VPL];
#pragma unroll
    for (int k = 0; k < VPL; ++k) {
        vlive[k] = kExact || (g < G && v + 32 * k < c.row_vecs);
        vzero[k] = zero_row + (v + 32 * k) % 128;
    }

    // Segment-end window: lane i holds the (relative) end of segment win + i.
    int32_t win = c.first;
    int32_t my_end = (win + lane < c.seg_hi) ? rel_pos(pol.seg_end(win + lane), c.k0) : kRelHi;
    int32_t seg = c.first;
    int32_t s_cur = kRelHi, e_cur = kRelHi;
    if (seg < c.seg_hi) {
        s_cur = rel_pos(pol.seg_begin(seg), c.k0);
        e_cur = __shfl_sync(kFull, my_end, 0);
    }

    // fp32 rows (tables or gradients) sum in two levels (see the fold below);
    // half-precision rows, whose tolerance is far looser, use one level, which
    // frees registers for occupancy.
    constexpr bool kTwoLevel = Pol::kTwoLevel;
    float ain[VPL][E], aout[VPL][kTwoLevel ? E : 1];
#pragma unroll
    for (int k = 0; k < VPL; ++k) {
#pragma unroll
        for (int x = 0; x < E; ++x) ain[k][x] = 0.f;
#pragma unroll
        for (int x = 0; x < (kTwoLevel ? E : 1); ++x) aout[k][x] = 0.f;
    }

    auto flush = [&]() {
        float tot[VPL][E];
#pragma unroll
        for (int k = 0; k < VPL; ++k)
#pragma unroll
            for (int x = 0; x < E; ++x) tot[k][x] = kTwoLevel ? aout[k][x] + ain[k][x] : ain[k][x];
        for (int off = V; off < V * G; off <<= 1) {
#pragma unroll
            for (int k = 0; k < VPL; ++k)
#pragma unroll
                for (int x = 0; x < E; ++x) tot[k][x] += __shfl_xor_sync(kFull, tot[k][x], off);
        }
        pol.emit(seg, e_cur - s_cur, s_cur >= 0, e_cur <= len, tot, v, g == 0);
#pragma unroll
        for (int k = 0; k < VPL; ++k) {
#pragma unroll
            for (int x = 0; x < E; ++x) ain[k][x] = 0.f;
#pragma unroll
            for (int x = 0; x < (kTwoLevel ? E : 1); ++x) aout[k][x] = 0.f;
        }
    };
    auto advance = [&]() {
        ++seg;
        s_cur = e_cur;
        if (seg >= c.seg_hi) {
            s_cur = e_cur = kRelHi;
            return;
        }
        if (seg - win >= 32) {
            win = seg;
            my_end = (win + lane < c.seg_hi) ? rel_pos(pol.seg_end(win + lane), c.k0) : kRelHi;
        }
        e_cur = __shfl_sync(kFull, my_end, seg - win);
    };

    typename Pol::Raw nxt = Pol::none();
    if (lane < len) nxt = pol.fetch(c.k0 + lane);

    for (int32_t base = 0; base < len; base += 32) {
        const int nb = min(32, len - base);
        const typename Pol::Raw cur = nxt;
        // Prefetch the next batch's raw payload while this batch's rows are in
        // flight; it is only decoded when its batch comes up.
        nxt = Pol::none();
        if (base + 32 + lane < len) nxt = pol.fetch(c.k0 + base + 32 + lane);
        uint32_t my_a = kInvalid;  // lanes >= nb hold kInvalid
        float my_w = 0.f;
        if (lane < nb) pol.decode(cur, my_a, my_w);

        for (int i0 = 0; i0 < nb; i0 += step) {
            // Issue every row load of the step first; an invalid or padding item
            // reads the zero row, so it adds nothing and needs no bookkeeping.
            uint4 buf[U][VPL];
            float wt[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int i = i0 + u * G + g;
                const uint32_t a = __shfl_sync(kFull, my_a, i & 31);
                wt[u] = W ? __shfl_sync(kFull, my_w, i & 31) : 1.f;
                const bool ok = u < ustop && a != kInvalid;
                const uint4* rp = pol.base + static_cast<size_t>(a) * pol.stride;
#pragma unroll
                for (int k = 0; k < VPL; ++k)
                    buf[u][k] = __ldg((ok && vlive[k]) ? rp + v + 32 * k : vzero[k]);
            }
            // Then add them in position order, emitting segments as they end.
            if (i0 + step <= nb && e_cur > base + i0 + step - 1) {
                // Common case: a full step inside the current segment.
#pragma unroll
                for (int u = 0; u < U; ++u)
#pragma unroll
                    for (int k = 0; k < VPL; ++k) accumulate<Pol::kDtype, W>(ain[k], buf[u][k], wt[u]);
                continue;
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int ifirst = i0 + u * G;
                if (ifirst >= nb) break;
                const int32_t qlast = base + min(ifirst + G, nb) - 1;  // last item of this row group
                if (e_cur > qlast) {
#pragma unroll
                    for (int k = 0; k < VPL; ++k) accumulate<Pol::kDtype, W>(ain[k], buf[u][k], wt[u]);
                } else {
                    // One or more segments end inside this row group.
                    const int32_t q = base + ifirst + g;
                    bool added = false;
                    do {
                        if (!added && q < e_cur) {
#pragma unroll
                            for (int k = 0; k < VPL; ++k)
                                accumulate<Pol::kDtype, W>(ain[k], buf[u][k], wt[u]);
                            added = true;
                        }
                        flush();
                        advance();
                    } while (e_cur <= qlast);
                    if (!added) {
#pragma unroll
                        for (int k = 0; k < VPL; ++k) accumulate<Pol::kDtype, W>(ain[k], buf[u][k], wt[u]);
                    }
                }
            }
        }
        // Two-level summation: at most 32 / G terms per lane enter `ain` before
        // it is folded into `aout`, which bounds the fp32 rounding error.
        if (kTwoLevel) {
#pragma unroll
            for (int k = 0; k < VPL; ++k)
#pragma unroll
                for (int x = 0; x < E; ++x) {
                    aout[k][x] += ain[k][x];
                    ain[k][x] = 0.f;
                }
        }
    }

    // Segments still open at the chunk end: finish those that end here, emit the
    // piece of the one that continues, and (last chunk only) the trailing empties.
    while (seg < c.seg_hi) {
        if (!c.last && s_cur >= len) break;
        const bool done = e_cur <= len;
        flush();
        if (!done) break;
        advance();
    }
}

// ---------------------------------------------------------------- the row walker
//
// walk_rows has walk_chunk's contract for the common layout, one 16-byte vector
// per lane and G = 32 / V rows per warp step fixed at compile time, and is built
// around batches of 32 item positions. Before a batch's rows are loaded, the
// warp finds every segment ending inside the batch from a window of 32 segment
// ends (one per lane): the positions of those ends become a 32-bit mask, and
// their segment numbers go to a per-warp list in shared memory, in order. Adding
// a row then costs a shuffle, one multiply-add for its address, the load and
// the adds, and the mask is tested once per group of loads; a segment end costs
// one list read and the store of the sum. Empty segments (empty bags) are
// written out during the scan. Pol additionally supplies:
//   static constexpr bool kEmptySegments    segments may be empty
//   static constexpr bool kUnrollGroups     unroll a batch's load groups
//   static constexpr bool kFastBatch        separate unrolled path for batches
//                                            with no segment end
//   static constexpr int kPrefetch          load groups ahead whose rows are
//                                            prefetched into L1 (0: none)
//   void put(seg, len, started, ends, tot, v, is_group0)   emit without the
//                                            per-segment metadata
//   void seg_meta(seg)                       metadata of a segment that began in
//                                            this chunk (once per segment; lanes
//                                            may call it for different segments
//                                            at the same time)
//   void put_empty(seg, v, is_group0)        the output of an empty segment

struct EndSlot {
    int32_t seg;
    int32_t len;  // segment length, or -1 when it began in an earlier chunk
};

// Loads of rows staged in shared memory (D > 0): each group of UG row steps is
// copied with cp.async into a per-warp ring of D + 1 groups of slots (16 bytes
// per lane and step), D groups ahead of the one being added, so that D * UG
// steps of rows are in flight per warp without holding registers. A slot is
// refilled one group after it was read, when its values have been added. The
// decoded payloads of the next batch are kept for the prefetch across the
// batch boundary. D = 0: the rows are loaded into registers one group at a
// time.
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 16;\n" ::"r"(
                     static_cast<uint32_t>(__cvta_generic_to_shared(smem))),
                 "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp_async8(void* smem, const void* gmem) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(
                     static_cast<uint32_t>(__cvta_generic_to_shared(smem))),
                 "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp_async4(void* smem, const void* gmem) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(
                     static_cast<uint32_t>(__cvta_generic_to_shared(smem))),
                 "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;\n" ::: "memory"); }

// A row's cache lines requested into L1 ahead of its load, without a register.
__device__ __forceinline__ void prefetch_l1(const void* p) {
    asm volatile("prefetch.global.L1 [%0];" ::"l"(p));
}

// KS > 0 (with D = 0): the items' raw payloads (indices and weights, or
// sorted payloads) are staged with cp.async KS batches ahead into a per-warp
// ring of KS + 1 batch slots (Pol::kStageBytes per lane), instead of being
// loaded into registers one batch ahead.
template <class Pol, int G, int D = 0, int KS = 0>
__device__ __forceinline__ void walk_rows(Pol& pol, const ChunkCtx& c, const uint4* zero_row,
                                          int lane, EndSlot* slots, uint4* ring = nullptr,
                                          char* stage = nullptr) {
    static_assert(G == 1 || G == 2 || G == 4 || G == 8, "rows per warp step");
    static_assert(Pol::kVpl == 1, "one vector per lane");
    constexpr int E = Pol::kElems;
    constexpr int V = 32 / G;
    constexpr int kSteps = 32 / G;                                      // row steps per batch
    constexpr int UG = Pol::kUnroll < kSteps ? Pol::kUnroll : kSteps;  // row steps per load group
    constexpr int kGroupItems = UG * G;
    constexpr uint32_t kGroupMask = kGroupItems == 32 ? kFull : (1u << kGroupItems) - 1u;
    constexpr uint32_t kStepMask = (1u << G) - 1u;
    constexpr bool W = Pol::kWeighted;
    constexpr bool kTwoLevel = Pol::kTwoLevel;
    constexpr int kGroupUnroll = Pol::kUnrollGroups ? 32 / kGroupItems : 1;
    const int g = lane / V;
    const int v = lane - g * V;
    const int32_t len = c.len;
    const char* lane_base = reinterpret_cast<const char*>(pol.base + v);
    const uint32_t row_bytes = pol.stride * 16u;
    const uint4* zrow = zero_row + v;
    const uint32_t below = (1u << lane) - 1u;

    float ain[E], aout[kTwoLevel ? E : 1];
#pragma unroll
    for (int x = 0; x < E; ++x) ain[x] = 0.f;
#pragma unroll
    for (int x = 0; x < (kTwoLevel ? E : 1); ++x) aout[x] = 0.f;

    // Window: lane j holds the relative end of segment seg + j.
    int32_t seg = c.first;
    int32_t s_cur = seg < c.seg_hi ? rel_pos(pol.seg_begin(seg), c.k0) : kRelHi;
    int32_t my_end = seg + lane < c.seg_hi ? rel_pos(pol.seg_end(seg + lane), c.k0) : kRelHi;
    uint32_t mask = 0;
    int ce_async = 0;  // next entry of the segment-end list (staged loads)

    // Segments ending at or before `bend` (the batch starts at `base`) leave the
    // window: non-empty ones are listed and marked in `mask`, empty ones owned
    // by this chunk are written out. Ends are non-decreasing, so the finished
    // segments are a prefix of the window.
    auto scan = [&](int32_t base, int32_t bend) {
        __syncwarp();  // every lane is done reading the previous batch's list
        mask = 0;
        int nend = 0;
        for (;;) {
            int32_t my_beg = __shfl_up_sync(kFull, my_end, 1);
            if (lane == 0) my_beg = s_cur;
            const bool nonempty = my_end > my_beg;
            const bool done = my_end <= bend && (nonempty || my_end < len || c.last);
            const uint32_t dm = __ballot_sync(kFull, done);
            const uint32_t ne = __ballot_sync(kFull, done && nonempty);
            if (done && nonempty) {
                // (index masked: malformed offsets, which are reported, can
                // break the prefix property but never reach past the list)
                slots[(nend + __popc(ne & below)) & 31] = EndSlot{seg + lane, my_beg >= 0 ? my_end - my_beg : -1};
                if (my_beg >= 0) pol.seg_meta(seg + lane);
            }
            if constexpr (Pol::kEmptySegments) {
                for (uint32_t em = dm & ~ne; em; em &= em - 1) pol.put_empty(seg + __ffs(em) - 1, v, g == 0);
            }
            mask |= __reduce_or_sync(kFull, (done && nonempty) ? 1u << ((my_end - base - 1) & 31) : 0u);
            nend += __popc(ne);
            const int nd = __popc(dm);
            if (nd == 0) break;
            const int32_t last_end = __shfl_sync(kFull, my_end, nd - 1);
            const int32_t moved = __shfl_down_sync(kFull, my_end, nd & 31);
            s_cur = last_end;
            seg += nd;
            my_end = lane + nd < 32 ? moved
                                    : (seg + lane < c.seg_hi ? rel_pos(pol.seg_end(seg + lane), c.k0) : kRelHi);
            // A full window that finished before `bend` leaves more to find; at
            // the chunk end, so may one that finished exactly there (empty
            // segments at the end of the table's last chunk).
            if (nd < 32 || (last_end >= bend && !(Pol::kEmptySegments && bend == len))) break;
        }
        __syncwarp();
    };

    auto flush = [&](const EndSlot s, bool ends) {
        // Kept inside this chunk's segment range whatever the list holds.
        const int32_t sseg = min(max(s.seg, c.first), c.seg_hi - 1);
        float tot[1][E];
#pragma unroll
        for (int x = 0; x < E; ++x) tot[0][x] = kTwoLevel ? aout[x] + ain[x] : ain[x];
#pragma unroll
        for (int off = V; off < 32; off <<= 1)
#pragma unroll
            for (int x = 0; x < E; ++x) tot[0][x] += __shfl_xor_sync(kFull, tot[0][x], off);
        pol.put(sseg, s.len, s.len >= 0, ends, tot, v, g == 0);
#pragma unroll
        for (int x = 0; x < E; ++x) ain[x] = 0.f;
#pragma unroll
        for (int x = 0; x < (kTwoLevel ? E : 1); ++x) aout[x] = 0.f;
    };

    // One batch's rows: CLEAN = 32 valid items (no padding, no skipped item).
    auto rows = [&](auto clean_tag, uint32_t my_a, float my_w, int nb) {
        constexpr bool CLEAN = decltype(clean_tag)::value;
        int ce = 0;
#pragma unroll(kGroupUnroll)
        for (int i0 = 0; i0 < 32; i0 += kGroupItems) {
            if (!CLEAN && i0 >= nb) break;
            uint4 buf[UG];
            float wt[UG];
#pragma unroll
            for (int u = 0; u < UG; ++u) {
                const int src = i0 + u * G + g;
                const uint32_t a = __shfl_sync(kFull, my_a, src);
                wt[u] = W ? __shfl_sync(kFull, my_w, src) : 1.f;
                const uint4* p = reinterpret_cast<const uint4*>(lane_base + static_cast<uint64_t>(a) * row_bytes);
                buf[u] = __ldg(CLEAN || a != kInvalid ? p : zrow);
            }
            // The rows of the group kPrefetch groups ahead in this batch start
            // moving into L1 while this group's loads are waited for.
            if constexpr (Pol::kPrefetch > 0) {
                const int pf = i0 + Pol::kPrefetch * kGroupItems;
                if (pf < 32) {
#pragma unroll
                    for (int u = 0; u < UG; ++u) {
                        const uint32_t a = __shfl_sync(kFull, my_a, pf + u * G + g);
                        if (a != kInvalid) prefetch_l1(lane_base + static_cast<uint64_t>(a) * row_bytes);
                    }
                }
            }
            const uint32_t m = (mask >> i0) & kGroupMask;
            if (m == 0) {
#pragma unroll
                for (int u = 0; u < UG; ++u) accumulate<Pol::kDtype, W>(ain, buf[u], wt[u]);
                continue;
            }
#pragma unroll
            for (int u = 0; u < UG; ++u) {
                uint32_t mu = (m >> (u * G)) & kStepMask;
                if (mu == 0) {
                    accumulate<Pol::kDtype, W>(ain, buf[u], wt[u]);
                    continue;
                }
                // Segments end after item i0 + u*G + p for each set bit p; this
                // group's item (p index g) belongs to the first of them with g <= p.
                bool added = false;
                do {
                    const int p = __ffs(mu) - 1;
                    if (!added && g <= p) {
                        accumulate<Pol::kDtype, W>(ain, buf[u], wt[u]);
                        added = true;
                    }
                    flush(slots[ce++], true);
                    mu &= mu - 1;
                } while (mu);
                if (!added) accumulate<Pol::kDtype, W>(ain, buf[u], wt[u]);
            }
        }
    };

    if constexpr (D > 0) {
        constexpr int kGroups = 32 / kGroupItems;  // load groups per batch
        // groups in flight: at most a batch's, so the prefetch reaches at most
        // one batch ahead
        constexpr int DD = D < kGroups ? D : kGroups;
        constexpr int kRing = DD + 1;              // groups of slots in the ring
        // The rows of load group q (0 .. kGroups-1) of a batch whose decoded
        // row numbers are `aa` and first position `bbase` go to ring group `rg`.
        auto issue = [&](int rg, uint32_t aa, int q, int32_t bbase) {
#pragma unroll
            for (int u = 0; u < UG; ++u) {
                const int src = q * kGroupItems + u * G + g;
                const uint32_t a = __shfl_sync(kFull, aa, src);
                const char* p = (a != kInvalid && bbase + src < len)
                                    ? lane_base + static_cast<uint64_t>(a) * row_bytes
                                    : reinterpret_cast<const char*>(zrow);
                cp_async16(ring + (rg * UG + u) * 32 + lane, p);
            }
            cp_async_commit();
        };
        // Decoded payloads of this batch and the next; raw payloads two ahead.
        uint32_t a0 = kInvalid, a1 = kInvalid;
        float w0 = 0.f, w1 = 0.f;
        typename Pol::Raw raw = Pol::none();
        if (lane < len) raw = pol.fetch(c.k0 + lane);
        if (lane < len) pol.decode(raw, a0, w0);
        raw = Pol::none();
        if (32 + lane < len) raw = pol.fetch(c.k0 + 32 + lane);
#pragma unroll
        for (int q = 0; q < DD; ++q) issue(q, a0, q, 0);
        int rd = 0;  // ring group read next
        for (int32_t base = 0; base < len; base += 32) {
            const int nb = min(32, len - base);
            a1 = kInvalid;
            w1 = 0.f;
            if (base + 32 + lane < len) pol.decode(raw, a1, w1);
            raw = Pol::none();
            if (base + 64 + lane < len) raw = pol.fetch(c.k0 + base + 64 + lane);
            scan(base, base + nb);
            for (int q = 0; q < kGroups; ++q) {
                if (base + q * kGroupItems >= len) {
                    // past the chunk: the groups still in flight carry zeros
                    continue;
                }
                cp_async_wait<DD - 1>();
                uint4 buf[UG];
                float wt[UG];
#pragma unroll
                for (int u = 0; u < UG; ++u) {
                    buf[u] = ring[(rd * UG + u) * 32 + lane];
                    wt[u] = W ? __shfl_sync(kFull, w0, q * kGroupItems + u * G + g) : 1.f;
                }
                // refill the ring group read one group ago with group q + DD
                const int wr = rd == 0 ? kRing - 1 : rd - 1;
                if (q + DD < kGroups) issue(wr, a0, q + DD, base);
                else issue(wr, a1, q + DD - kGroups, base + 32);
                rd = rd + 1 == kRing ? 0 : rd + 1;
                const uint32_t m = (mask >> (q * kGroupItems)) & kGroupMask;
                if (m == 0) {
#pragma unroll
                    for (int u = 0; u < UG; ++u) accumulate<Pol::kDtype, W>(ain, buf[u], wt[u]);
                    continue;
                }
#pragma unroll
                for (int u = 0; u < UG; ++u) {
                    uint32_t mu = (m >> (u * G)) & kStepMask;
                    if (mu == 0) {
                        accumulate<Pol::kDtype, W>(ain, buf[u], wt[u]);
                        continue;
                    }
                    bool added = false;
                    do {
                        const int p = __ffs(mu) - 1;
                        if (!added && g <= p) {
                            accumulate<Pol::kDtype, W>(ain, buf[u], wt[u]);
                            added = true;
                        }
                        flush(slots[ce_async++], true);
                        mu &= mu - 1;
                    } while (mu);
                    if (!added) accumulate<Pol::kDtype, W>(ain, buf[u], wt[u]);
                }
            }
            ce_async = 0;
            if (kTwoLevel) {
#pragma unroll
                for (int x = 0; x < E; ++x) {
                    aout[x] += ain[x];
                    ain[x] = 0.f;
                }
            }
            a0 = a1;
            w0 = w1;
        }
        cp_async_wait_all();
        __syncwarp();
        scan(len, len);
        if (seg < c.seg_hi && s_cur < len) {
            if (s_cur >= 0 && lane == 0) pol.seg_meta(seg);
            flush(EndSlot{seg, s_cur >= 0 ? 0 : -1}, false);
        }
        return;
    }

    typename Pol::Raw nxt = Pol::none();
    constexpr int kStage = KS > 0 ? KS : 1;
    auto stage_slot = [&](int k) { return stage + (k * 32 + lane) * Pol::kStageBytes; };
    int srd = 0;  // staging slot of the batch read next
    if constexpr (KS > 0) {
#pragma unroll
        for (int k = 0; k < kStage; ++k) {
            if (k * 32 + lane < len) pol.stage(stage_slot(k), c.k0 + k * 32 + lane);
            cp_async_commit();
        }
    } else {
        if (lane < len) nxt = pol.fetch(c.k0 + lane);
    }
    for (int32_t base = 0; base < len; base += 32) {
        const int nb = min(32, len - base);
        typename Pol::Raw cur = nxt;
        if constexpr (KS > 0) {
            cp_async_wait<kStage - 1>();
            cur = lane < nb ? pol.staged(stage_slot(srd)) : Pol::none();
            // refill the slot read one batch ago with the batch KS ahead
            const int swr = srd == 0 ? kStage : srd - 1;
            if (base + kStage * 32 + lane < len) pol.stage(stage_slot(swr), c.k0 + base + kStage * 32 + lane);
            cp_async_commit();
            srd = srd == kStage ? 0 : srd + 1;
        } else {
            nxt = Pol::none();
            if (base + 32 + lane < len) nxt = pol.fetch(c.k0 + base + 32 + lane);
        }
        uint32_t my_a = kInvalid;
        float my_w = 0.f;
        if (lane < nb) pol.decode(cur, my_a, my_w);
        scan(base, base + nb);
        const bool clean = __all_sync(kFull, my_a != kInvalid);
        if (Pol::kFastBatch && clean && mask == 0) {
            // The whole batch adds into the open segment: every load group
            // unrolled, so loads of later groups overlap the adds of earlier ones.
#pragma unroll
            for (int i0 = 0; i0 < 32; i0 += kGroupItems) {
#pragma unroll
                for (int u = 0; u < UG; ++u) {
                    const int src = i0 + u * G + g;
                    const uint32_t a = __shfl_sync(kFull, my_a, src);
                    const float w = W ? __shfl_sync(kFull, my_w, src) : 1.f;
                    const uint4 x = __ldg(reinterpret_cast<const uint4*>(
                        lane_base + static_cast<uint64_t>(a) * row_bytes));
                    accumulate<Pol::kDtype, W>(ain, x, w);
                }
            }
        } else if (clean) {
            rows(std::true_type{}, my_a, my_w, nb);
        } else {
            rows(std::false_type{}, my_a, my_w, nb);
        }
        // Two-level summation: at most 32 / G terms per lane enter `ain` before
        // it is folded into `aout`, which bounds the fp32 rounding error.
        if (kTwoLevel) {
#pragma unroll
            for (int x = 0; x < E; ++x) {
                aout[x] += ain[x];
                ain[x] = 0.f;
            }
        }
    }
    if constexpr (KS > 0) {
        cp_async_wait_all();
        __syncwarp();
    }
    // Empty segments at the chunk end (last chunk of a table), and chunks with
    // no items; then the piece of the segment that runs past the chunk end.
    scan(len, len);
    if (seg < c.seg_hi && s_cur < len) {
        if (s_cur >= 0 && lane == 0) pol.seg_meta(seg);
        flush(EndSlot{seg, s_cur >= 0 ? 0 : -1}, false);
    }
}

// ---------------------------------------------------------------- fix-up

// A segment that straddles chunks left its tail piece in chunk j and head pieces
// in the m chunks after it (chunks of a table are contiguous and chunk_len long
// except the table's last, so m follows from the segment end). The pieces are
// added in a fixed order, so the result is deterministic; `store` receives each
// group of four columns in fp64. Up to 32 pieces: lanes own columns and walk the
// pieces (add_pieces); more pieces (a hot row repeated across hundreds of
// chunks): lanes own pieces and meet in a butterfly per group of four columns.
constexpr int kInnerPieces = 16;

// acc (fp64, four columns from x0) += pieces i0, i0 + step, ... below m, each at
// head + piece * dmax. The pieces are summed in fp32 in groups of kInnerPieces,
// each group folded into acc: GB300's fp64 adds are scarce (one per piece and
// column made a heavy-run combine fp64-bound), and an fp32 sum of at most 16
// pieces rounds within 16u of their absolute sum. Four loads in flight.
__device__ __forceinline__ void add_pieces(const float* head, int64_t i0, int64_t step, int64_t m, int dmax,
                                           int x0, double (&acc)[4]) {
    for (int64_t g = i0; g < m; g += kInnerPieces * step) {
        const int64_t gend = min64(m, g + kInnerPieces * step);
        float in[4] = {0.f, 0.f, 0.f, 0.f};
        int64_t i = g;
        for (; i + 3 * step < gend; i += 4 * step) {
            float4 h[4];
#pragma unroll
            for (int c = 0; c < 4; ++c) h[c] = *reinterpret_cast<const float4*>(head + (i + c * step) * dmax + x0);
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                in[0] += h[c].x;
                in[1] += h[c].y;
                in[2] += h[c].z;
                in[3] += h[c].w;
            }
        }
        for (; i < gend; i += step) {
            const float4 h = *reinterpret_cast<const float4*>(head + i * dmax + x0);
            in[0] += h.x;
            in[1] += h.y;
            in[2] += h.z;
            in[3] += h.w;
        }
#pragma unroll
        for (int x = 0; x < 4; ++x) acc[x] += in[x];
    }
}

template <class Store>
__device__ __forceinline__ void combine_pieces(const Plan& Q, int64_t j, int64_t m, int dim,
                                               int dmax, int lane, Store store) {
    const float* tail = Q.carry_tail + j * dmax;
    const float* head = Q.carry_head + (j + 1) * dmax;
    if (m <= 32) {
        for (int x0 = lane * 4; x0 < dim; x0 += 128) {
            const float4 a = *reinterpret_cast<const float4*>(tail + x0);
            double acc[4] = {a.x, a.y, a.z, a.w};
            add_pieces(head, 0, 1, m, dmax, x0, acc);
            store(x0, acc);
        }
        return;
    }
    // Four groups of four columns per round: 16 independent loads per lane.
    for (int x0 = 0; x0 < dim; x0 += 16) {
        double acc[4][4] = {};
        const int ng = min(4, (dim - x0) / 4);
        if (lane == 0) {
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                if (c >= ng) break;
                const float4 a = *reinterpret_cast<const float4*>(tail + x0 + 4 * c);
                acc[c][0] = a.x;
                acc[c][1] = a.y;
                acc[c][2] = a.z;
                acc[c][3] = a.w;
            }
        }
#pragma unroll 4
        for (int64_t i = lane; i < m; i += 32) {
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                if (c >= ng) break;
                const float4 h = *reinterpret_cast<const float4*>(head + i * dmax + x0 + 4 * c);
                acc[c][0] += h.x;
                acc[c][1] += h.y;
                acc[c][2] += h.z;
                acc[c][3] += h.w;
            }
        }
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1)
#pragma unroll
            for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int x = 0; x < 4; ++x) acc[c][x] += __shfl_xor_sync(kFull, acc[c][x], off);
        if (lane == 0) {
#pragma unroll
            for (int c = 0; c < 4; ++c)
                if (c < ng) store(x0 + 4 * c, acc[c]);
        }
    }
}

// Number of chunks after chunk j that a segment ending at `e` reaches into.
__device__ __forceinline__ int64_t pieces_after(const Plan& Q, int64_t j, int64_t e, int64_t total) {
    const Chunk ch = Q.chunks[j];
    const int64_t k1 = ch.k0 + static_cast<int64_t>(ch.len & 0x7fffffffu);
    if (e <= k1) return 0;
    const int64_t m = (e - k1 + Q.chunk_len - 1) / Q.chunk_len;
    return min64(m, total - j - 1);
}

// ---------------------------------------------------------------- small scans

// Inclusive warp scan.
__device__ __forceinline__ int64_t warp_incl_scan(int64_t x, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int64_t y = __shfl_up_sync(kFull, x, o);
        if (lane >= o) x += y;
    }
    return x;
}

// Exclusive block scan for blockDim.x a multiple of 32 (<= 1024). `sh` needs
// 33 int64 slots. Returns the exclusive prefix; *total receives the block sum.
__device__ __forceinline__ int64_t block_excl_scan(int64_t x, int64_t* sh, int64_t* total) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
    const int64_t inc = warp_incl_scan(x, lane);
    if (lane == 31) sh[wid] = inc;
    __syncthreads();
    if (wid == 0) {
        int64_t s = lane < nw ? sh[lane] : 0;
        const int64_t si = warp_incl_scan(s, lane);
        if (lane < nw) sh[lane] = si - s;
        if (lane == 31) sh[32] = si;
    }
    __syncthreads();
    const int64_t r = sh[wid] + inc - x;
    *total = sh[32];
    __syncthreads();
    return r;
}

}  // namespace cbtbe
