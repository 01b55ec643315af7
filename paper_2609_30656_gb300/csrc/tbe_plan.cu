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

// mode 0: first = the bag touching the chunk start (forward, key generation).
// mode 1: first = the run of sorted ids containing the chunk start (reduce).
// mode 2: tiles only (radix sort), first left at 0.
__global__ void plan_chunks_kernel(Problem P, Plan Q, int mode, const uint32_t* seg_start,
                                   const int64_t* num_unique) {
    const int64_t total = min(Q.class_chunk_base[Q.num_classes], Q.max_chunks);
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    const int64_t C = Q.chunk_len;
    const int64_t U = mode == 1 ? *num_unique : 0;
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
        const int64_t p1 = max(p0, Q.table_pos[t + 1]);
        const int64_t nch = max(static_cast<int64_t>(1), (p1 - p0 + C - 1) / C);
        const int64_t k0 = min(p0 + local * C, p1);
        const int64_t len = min(C, p1 - k0);
        const bool last = local >= nch - 1;
        int64_t first = 0;
        if (mode == 2) {
            // tiles only (radix sort): no first segment needed
        } else if (mode == 0) {
            // First bag b of table t with offsets[b] >= k0 (lower bound over the
            // table's B + 1 offsets); the chunk starts in the bag before it unless
            // a bag starts exactly at k0.
            const int64_t blo = static_cast<int64_t>(t) * P.B, bhi = blo + P.B;
            int64_t a = blo, b = bhi + 1;
            while (a < b) {
                const int64_t m = (a + b) >> 1;
                if (load_index(P.offsets, m, P.is32) < k0) a = m + 1; else b = m;
            }
            first = (a <= bhi && load_index(P.offsets, a, P.is32) == k0) ? a : a - 1;
            first = min(max(first, blo), bhi);
        } else {
            // Last run u with seg_start[u] <= k0.
            int64_t a = 0, b = U + 1;
            while (a < b) {
                const int64_t m = (a + b) >> 1;
                if (static_cast<int64_t>(seg_start[m]) <= k0) a = m + 1; else b = m;
            }
            first = max(a - 1, static_cast<int64_t>(0));
        }
        Chunk ch;
        ch.k0 = k0;
        ch.first = first;
        ch.table = t;
        ch.len = static_cast<uint32_t>(len) | (last ? 0x80000000u : 0u);
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
