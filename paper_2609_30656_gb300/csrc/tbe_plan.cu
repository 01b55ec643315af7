// tbe_plan.cu -- offsets validation and the chunk plan shared by the forward
// gather-pool and the backward key generation / segmented reduce.
//
// A table's items (lookup positions, key-major so each table's lookups are
// contiguous) are cut into chunks of at most chunk_len positions; a table with
// no lookups still gets one (empty) chunk so that its empty bags are written.
// Chunks are numbered class by class (tables grouped by kernel instantiation),
// table by table within a class.
#include "tbe_internal.cuh"
#include "tbe_launch.h"

namespace cbtbe {

__global__ void validate_offsets_kernel(Problem P) {
    const int64_t nb = static_cast<int64_t>(P.T) * P.B;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t k = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; k <= nb;
         k += stride) {
        const int64_t o = load_index(P.offsets, k, P.is32);
        bool bad = o < 0 || o > P.n;
        if (k == 0 && o != 0) bad = true;
        if (k == nb && o != P.n) bad = true;
        if (k < nb && load_index(P.offsets, k + 1, P.is32) < o) bad = true;
        if (bad) set_error(P.error, CB_ERR_BAD_OFFSETS);
    }
}

// One block: table item ranges, then per class a scan of the tables' chunk counts.
__global__ void __launch_bounds__(1024) plan_tables_kernel(Problem P, Plan Q) {
    __shared__ int64_t sh[33];
    __shared__ int64_t running;
    const int tid = threadIdx.x;
    for (int t = tid; t <= P.T; t += blockDim.x) {
        int64_t pos = load_index(P.offsets, static_cast<int64_t>(t) * P.B, P.is32);
        Q.table_pos[t] = min(max(pos, static_cast<int64_t>(0)), P.n);
    }
    if (tid == 0) running = 0;
    __syncthreads();
    const int64_t C = Q.chunk_len;
    for (int c = 0; c < Q.num_classes; ++c) {
        if (tid == 0) Q.class_chunk_base[c] = min(running, Q.max_chunks);
        const int a = Q.class_table_start[c], b = Q.class_table_start[c + 1];
        for (int i0 = a; i0 < b; i0 += blockDim.x) {
            const int i = i0 + tid;
            int64_t cnt = 0;
            if (i < b) {
                const int t = Q.class_tables[i];
                const int64_t nt = max(static_cast<int64_t>(0), Q.table_pos[t + 1] - Q.table_pos[t]);
                cnt = max(static_cast<int64_t>(1), (nt + C - 1) / C);
            }
            int64_t total;
            const int64_t ex = block_excl_scan(cnt, sh, &total);
            if (i < b) Q.ord_chunk_base[i] = running + ex;
            __syncthreads();
            if (tid == 0) running += total;
            __syncthreads();
        }
    }
    if (tid == 0) {
        Q.class_chunk_base[Q.num_classes] = min(running, Q.max_chunks);
        Q.ord_chunk_base[P.T] = running;
        if (running > Q.max_chunks) set_error(P.error, CB_ERR_BAD_OFFSETS);
    }
}

// Segment bounds around a position: the first bag of table t starting at or
// after x (lower bound over the table's offsets), or the run of sorted ids
// containing x.
__device__ __forceinline__ int64_t bag_lower_bound(const Problem& P, int t, int64_t x) {
    const int64_t blo = static_cast<int64_t>(t) * P.B, bhi = blo + P.B;
    int64_t a = blo, b = bhi + 1;
    while (a < b) {
        const int64_t m = (a + b) >> 1;
        if (load_index(P.offsets, m, P.is32) < x) a = m + 1; else b = m;
    }
    return a;  // in [blo, bhi + 1]
}

__device__ __forceinline__ int64_t run_containing(const uint32_t* seg_start, int64_t U, int64_t x) {
    int64_t a = 0, b = U + 1;
    while (a < b) {
        const int64_t m = (a + b) >> 1;
        if (static_cast<int64_t>(seg_start[m]) <= x) a = m + 1; else b = m;
    }
    return max64(a - 1, 0);
}

// A chunk boundary at x moves to the end of the segment it falls in, unless
// that segment is longer than the cap: short bags and runs are then never
// split, and only heavy ones leave pieces for the fix-up. Monotone in x, so
// consecutive chunks stay contiguous (a chunk may come out empty). One search
// gives both the moved boundary and the first segment of a chunk starting
// there:
//   mode 0: the bag touching the chunk start (the bag starting exactly there if
//           any, the first of equal starts; else the one containing it);
//   mode 1: the run of sorted ids containing the chunk start;
//   mode 2: tiles only (radix sort), no moving, first left at 0.
struct Boundary {
    int64_t k;      // position
    int64_t first;  // first segment of a chunk starting at k
};

__device__ __forceinline__ Boundary boundary(const Problem& P, const Plan& Q, int mode, int t,
                                             const uint32_t* seg_start, int64_t U, int64_t x, int64_t p0,
                                             int64_t p1) {
    const bool may_move = Q.snap_cap > 0 && x > p0 && x < p1;
    if (mode == 0) {
        const int64_t blo = static_cast<int64_t>(t) * P.B, bhi = blo + P.B;
        const int64_t a = bag_lower_bound(P, t, x);  // first bag starting at or after x
        const int64_t e = a <= bhi ? load_index(P.offsets, a, P.is32) : -1;
        int64_t k = x;
        if (may_move && a <= bhi && e != x && a != blo) {
            const int64_t s0 = load_index(P.offsets, a - 1, P.is32);
            if (e - s0 <= Q.snap_cap && e <= p1) k = e;
        }
        // Moved to e (= offsets[a], with offsets[a - 1] < x < e): bag a starts
        // there. Else the bag starting exactly at x, or the one containing it.
        const int64_t first = (a <= bhi && e == k) ? a : a - 1;
        return {k, min64(max64(first, blo), bhi)};
    }
    if (mode == 1) {
        const int64_t u = run_containing(seg_start, U, x);
        const int64_t s0 = seg_start[u], e = seg_start[u + 1];
        // Runs are never empty (seg_start increases), so the run containing e is u + 1.
        if (may_move && s0 != x && e - s0 <= Q.snap_cap && e <= p1) return {e, u + 1};
        return {x, u};
    }
    return {x, 0};
}

// 8 blocks of 256 threads per SM (32 registers): the grid (8 per SM) runs in
// one wave of latency-bound searches.
__global__ void __launch_bounds__(256, 8) plan_chunks_kernel(Problem P, Plan Q, int mode,
                                                             const uint32_t* seg_start,
                                                             const int64_t* num_unique) {
    const int64_t total = min64(Q.class_chunk_base[Q.num_classes], Q.max_chunks);
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    const int64_t C = Q.chunk_len;
    const int64_t U = mode == 1 ? *num_unique : 0;
    if (blockIdx.x == 0 && Q.chunk_next)  // the walkers' chunk counters (none for sort tiles)
        for (int c = threadIdx.x; c <= Q.num_classes; c += blockDim.x) Q.chunk_next[c] = 0;
    for (int64_t j = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; j < total;
         j += stride) {
        // Largest i with ord_chunk_base[i] <= j (each table has >= 1 chunk).
        int lo = 0, hi = P.T;
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (Q.ord_chunk_base[mid] <= j) lo = mid; else hi = mid;
        }
        const int t = Q.class_tables[lo];
        const int64_t local = j - Q.ord_chunk_base[lo];
        const int64_t p0 = Q.table_pos[t];
        const int64_t p1 = max64(p0, Q.table_pos[t + 1]);
        const int64_t nch = max64(1, (p1 - p0 + C - 1) / C);
        const bool last = local >= nch - 1;
        const int64_t x0 = min64(p0 + local * C, p1);
        const int64_t x1 = last ? p1 : min64(p0 + (local + 1) * C, p1);
        const Boundary b0 = boundary(P, Q, mode, t, seg_start, U, x0, p0, p1);
        const int64_t k1 = last ? x1 : boundary(P, Q, mode, t, seg_start, U, x1, p0, p1).k;
        Chunk ch;
        ch.k0 = b0.k;
        ch.first = b0.first;
        ch.table = t;
        ch.len = static_cast<uint32_t>(max64(0, k1 - b0.k)) | (last ? 0x80000000u : 0u);
        Q.chunks[j] = ch;
    }
}

void launch_validate_offsets(const Problem& P, int num_sms, cudaStream_t s) {
    const int64_t nb = static_cast<int64_t>(P.T) * P.B + 1;
    const int blocks = static_cast<int>(min64((nb + 255) / 256, int64_t(num_sms) * 8));
    validate_offsets_kernel<<<max(blocks, 1), 256, 0, s>>>(P);
}

void launch_plan(const Problem& P, const Plan& Q, int mode, const uint32_t* seg_start,
                 const int64_t* num_unique, int num_sms, bool tables_too, cudaStream_t s) {
    if (tables_too) plan_tables_kernel<<<1, 1024, 0, s>>>(P, Q);
    const int blocks = static_cast<int>(
        min64((Q.max_chunks + 255) / 256, static_cast<int64_t>(num_sms) * 8));
    plan_chunks_kernel<<<max(blocks, 1), 256, 0, s>>>(P, Q, mode, seg_start, num_unique);
}

}  // namespace cbtbe
