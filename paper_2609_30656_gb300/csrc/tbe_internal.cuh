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

#include "cb_tbe.h"

namespace cbtbe {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kWarpThreads = 256;  // block size of the warp-per-chunk kernels
constexpr int64_t kNoSeg = INT64_MAX;

// Per-table facts the kernels need, built once at create time.
struct TableDev {
    const void* data;   // row-major [rows, dim] of dtype
    int64_t rows;
    int64_t row_base;   // rows of all tables before this one (global row id base)
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
};

struct Plan {
    int32_t chunk_len;
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

// ---------------------------------------------------------------- the walker
//
// Pol (policy) supplies:
//   kElems, kVpl (16-byte vectors per lane), kUnroll (items in flight per lane)
//   int64_t seg_end(int64_t s)          end position of segment s (s < seg_hi)
//   void item(int64_t q, int64_t& a, float& w)   payload of item q (lane-local)
//   const uint4* row(int64_t a, bool& ok)         row of an item (ok=false: skip)
//   void unpack(const uint4&, float (&)[kElems])
//   void emit(seg, s, e, started, ends, tot, lane-in-group v, is_group0)
// The segment range of the chunk is [first, seg_hi); segments that start at or
// after the chunk end belong to the next chunk, except after the last chunk of a
// table (trailing empty bags), which `last` allows.

struct ChunkCtx {
    int64_t k0, k1;       // item positions [k0, k1)
    int64_t first;        // first segment
    int64_t seg_hi;       // segments of this table end before seg_hi
    int32_t lanes;        // V
    int32_t groups;       // G
    int32_t row_vecs;     // vectors per row
    bool last;            // owns trailing segments that start at k1
};

template <class Pol>
__device__ __forceinline__ void walk_chunk(Pol& pol, const ChunkCtx& c, int lane) {
    constexpr int E = Pol::kElems;
    constexpr int VPL = Pol::kVpl;
    constexpr int U = Pol::kUnroll;
    const int V = c.lanes, G = c.groups;
    const int g = lane / V;
    const int v = lane - g * V;
    const bool active = g < G;

    // Segment-end window: lane i holds the end of segment win_base + i.
    int64_t win_base = c.first;
    int64_t my_end = (win_base + lane < c.seg_hi) ? pol.seg_end(win_base + lane) : kNoSeg;
    int64_t seg = c.first;
    int64_t s_cur = kNoSeg, e_cur = kNoSeg;
    if (seg < c.seg_hi) {
        s_cur = pol.seg_begin(seg);
        e_cur = __shfl_sync(kFull, my_end, 0);
    }

    float ain[VPL][E], aout[VPL][E];
#pragma unroll
    for (int k = 0; k < VPL; ++k)
#pragma unroll
        for (int x = 0; x < E; ++x) ain[k][x] = aout[k][x] = 0.f;

    auto flush = [&]() {
        float tot[VPL][E];
#pragma unroll
        for (int k = 0; k < VPL; ++k)
#pragma unroll
            for (int x = 0; x < E; ++x) tot[k][x] = aout[k][x] + ain[k][x];
        for (int off = V; off < V * G; off <<= 1) {
#pragma unroll
            for (int k = 0; k < VPL; ++k)
#pragma unroll
                for (int x = 0; x < E; ++x) tot[k][x] += __shfl_xor_sync(kFull, tot[k][x], off);
        }
        pol.emit(seg, s_cur, e_cur, s_cur >= c.k0, e_cur <= c.k1, tot, v, g == 0);
#pragma unroll
        for (int k = 0; k < VPL; ++k)
#pragma unroll
            for (int x = 0; x < E; ++x) ain[k][x] = aout[k][x] = 0.f;
    };
    auto advance = [&]() {
        ++seg;
        s_cur = e_cur;
        if (seg >= c.seg_hi) {
            s_cur = e_cur = kNoSeg;
            return;
        }
        if (seg - win_base >= 32) {
            win_base = seg;
            my_end = (win_base + lane < c.seg_hi) ? pol.seg_end(win_base + lane) : kNoSeg;
        }
        e_cur = __shfl_sync(kFull, my_end, static_cast<int>(seg - win_base));
    };

    int64_t nxt_a = 0;
    float nxt_w = 1.f;
    if (c.k0 + lane < c.k1) pol.item(c.k0 + lane, nxt_a, nxt_w);

    for (int64_t base = c.k0; base < c.k1; base += 32) {
        const int nb = static_cast<int>(min64(32, c.k1 - base));
        const int64_t my_a = nxt_a;
        const float my_w = nxt_w;
        // Prefetch the next batch's payload while this batch's rows are in flight.
        nxt_a = 0;
        nxt_w = 1.f;
        if (base + 32 + lane < c.k1) pol.item(base + 32 + lane, nxt_a, nxt_w);

        for (int i0 = 0; i0 < nb; i0 += U * G) {
            uint4 buf[U][VPL];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int i = i0 + u * G + g;
                const int64_t a = __shfl_sync(kFull, my_a, i & 31);
                bool ok = active && i < nb;
                const uint4* rp = pol.row(a, ok);
#pragma unroll
                for (int k = 0; k < VPL; ++k) {
                    const int vec = v + k * 32;
                    buf[u][k] = (ok && vec < c.row_vecs) ? __ldg(rp + vec) : make_uint4(0, 0, 0, 0);
                }
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int ifirst = i0 + u * G;
                if (ifirst >= nb) break;
                const int i = ifirst + g;
                const float w = __shfl_sync(kFull, my_w, i & 31);
                const int64_t q = base + i;
                const int64_t qmax = base + min(ifirst + G, nb) - 1;
                bool added = !(active && i < nb);
                while (true) {
                    if (!added && q < e_cur) {
#pragma unroll
                        for (int k = 0; k < VPL; ++k) {
                            float f[E];
                            pol.unpack(buf[u][k], f);
#pragma unroll
                            for (int x = 0; x < E; ++x) ain[k][x] = fmaf(w, f[x], ain[k][x]);
                        }
                        added = true;
                    }
                    if (e_cur > qmax) break;
                    flush();
                    advance();
                }
            }
        }
        // Two-level summation: at most 32 / G terms per lane enter `ain` before
        // it is folded into `aout`, which bounds the fp32 rounding error.
#pragma unroll
        for (int k = 0; k < VPL; ++k)
#pragma unroll
            for (int x = 0; x < E; ++x) {
                aout[k][x] += ain[k][x];
                ain[k][x] = 0.f;
            }
    }

    // Segments still open at the chunk end: finish those that end here, emit the
    // piece of the one that continues, and (last chunk only) the trailing empties.
    while (seg < c.seg_hi) {
        if (!c.last && s_cur >= c.k1) break;
        const bool done = e_cur <= c.k1;
        flush();
        if (!done) break;
        advance();
    }
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
