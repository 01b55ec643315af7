// tbe_backward.cu -- de-duplicated backward of the pooled embedding bag with
// respect to the table rows (the adjoint of the sparse_arch lookup, Sec. IV.A.2):
//   G[row_base_t + r] = sum_{i : table t, indices[i] == r} w_i * s_b(i) * grad_out[b(i), Doff_t ..]
//
// Steps: (1) key generation: one warp per chunk of lookups walks the bags and
// writes key_i = key_base_t + indices[i] with a payload (the bag id, or the
// lookup position plus a packed (bag, w_i * s_b) pair when a coefficient is
// needed); (2) radix sort of each table's range;
// (3) run-length pass over the sorted ids; (4) per-table unique ranges and
// packed gradient offsets; (5) segmented reduce of the gathered grad_out
// slices, one warp per chunk of sorted positions; (6) fp64 fix-up of runs that
// straddle chunks.
#include <cuda_bf16.h>

#include "tbe_internal.cuh"
#include "tbe_launch.h"
#include "tbe_reduce.cuh"

namespace cbtbe {

constexpr int kRleThreads = 256;
constexpr int kRleItems = 16;
constexpr int kRleTile = kRleThreads * kRleItems;

// ---------------------------------------------------------------- (1) keys

// The bag of each lookup, from a window of 32 bag ends held one per lane, in
// positions relative to the chunk start: every position is below 2^30, so these
// are exact in 32 bits (saturated, for malformed offsets, well inside the
// sentinel kPastTable that marks ends past the table's last bag).
constexpr int32_t kPastTable = INT32_MAX;

__device__ __forceinline__ int32_t rel32(int64_t x, int64_t k0) {
    const int64_t r = x - k0;
    return static_cast<int32_t>(r < -(int64_t(1) << 30) ? -(int64_t(1) << 30)
                                                        : (r > (int64_t(1) << 30) ? (int64_t(1) << 30) : r));
}

struct BagWindow32 {
    int64_t win;        // first bag of the window
    int32_t win_start;  // start of bag win
    int32_t my_end;     // end of bag win + lane
};

__device__ __forceinline__ BagWindow32 bag_window32(const Problem& P, int64_t first, int64_t bag_hi,
                                                    int64_t k0, int lane) {
    BagWindow32 W;
    W.win = first;
    W.win_start = first < bag_hi ? rel32(load_index(P.offsets, first, P.is32), k0) : kPastTable;
    W.my_end = first + lane < bag_hi ? rel32(load_index(P.offsets, first + lane + 1, P.is32), k0) : kPastTable;
    return W;
}

// Every lane calls this with its relative position q; the window moves forward
// 32 bags at a time until every valid lane has its bag (bag = -1 otherwise).
__device__ __forceinline__ void find_bag32(const Problem& P, BagWindow32& W, int64_t bag_hi, int64_t k0,
                                           int32_t q, bool valid, int lane, int64_t& bag, int32_t& s,
                                           int32_t& e) {
    bag = -1;
    s = e = 0;
    while (true) {
        int cnt = 0;  // ends at or before q in the window
#pragma unroll
        for (int b = 16; b >= 1; b >>= 1)
            if (__shfl_sync(kFull, W.my_end, cnt + b - 1) <= q) cnt += b;
        if (__shfl_sync(kFull, W.my_end, 31) <= q) cnt = 32;
        const int32_t e_sel = __shfl_sync(kFull, W.my_end, cnt < 32 ? cnt : 31);
        const int32_t s_sel = __shfl_sync(kFull, W.my_end, cnt > 0 ? cnt - 1 : 0);
        if (valid && bag < 0 && cnt < 32) {
            bag = W.win + cnt;
            e = e_sel;
            s = cnt > 0 ? s_sel : W.win_start;
        }
        if (!__any_sync(kFull, valid && bag < 0)) break;
        W.win_start = __shfl_sync(kFull, W.my_end, 31);
        W.win += 32;
        W.my_end = W.win + lane < bag_hi ? rel32(load_index(P.offsets, W.win + lane + 1, P.is32), k0) : kPastTable;
    }
}

// The bags of 32 consecutive positions p0 .. p0 + 31 without shuffles when
// possible: the window's ends inside the step become bits of a mask (one warp
// OR), and lane l's bag is the window's first bag plus the ends at or before
// p0 + l. Returns false (nothing written) when two ends coincide (an empty bag)
// or the step reaches past the window's last end; the caller then bisects.
#ifndef CB_KEYGEN_MASK
#define CB_KEYGEN_MASK 1
#endif
__device__ __forceinline__ bool bags_by_mask(const BagWindow32& W, int32_t p0, int lane, bool want_range,
                                             int64_t& bag, int32_t& s, int32_t& e) {
    const bool before = W.my_end < p0;
    const bool inside = W.my_end >= p0 && W.my_end <= p0 + 31;
    const uint32_t nbefore = __popc(__ballot_sync(kFull, before));
    const uint32_t nin = __popc(__ballot_sync(kFull, inside));
    const uint32_t mask = __reduce_or_sync(kFull, inside ? 1u << (W.my_end - p0) : 0u);
    if (__popc(mask) != static_cast<int>(nin) || nbefore + nin >= 32) return false;  // warp-uniform
    const uint32_t le = lane == 31 ? kFull : (2u << lane) - 1u;
    const int cnt = static_cast<int>(nbefore) + __popc(mask & le);
    bag = W.win + cnt;
    if (want_range) {
        e = __shfl_sync(kFull, W.my_end, cnt);
        const int32_t prev = __shfl_sync(kFull, W.my_end, cnt > 0 ? cnt - 1 : 0);
        s = cnt > 0 ? prev : W.win_start;
    }
    return true;
}

// A warp walks one chunk kKeygenSteps x 32 lookups at a time: the indices (and
// weights) of all the steps are loaded first, so that many loads are in flight
// per warp, then each step finds its lanes' bags and writes.
#ifndef CB_KEYGEN_STEPS
#define CB_KEYGEN_STEPS 12
#endif
constexpr int kKeygenSteps = CB_KEYGEN_STEPS;

// Compiled with no minimum of resident blocks: 48 registers, 5 blocks of 256
// threads per SM. (A minimum of 1 let it take 72 registers, 3 blocks: cfg5
// 0.63 -> 0.75 ms; a minimum of 6, 40 registers: cfg5u 0.63 -> 0.71 ms.)
template <bool PACKED>
__global__ void __launch_bounds__(kWarpThreads) keygen_kernel(Problem P, Plan Q, KeyGen K) {
    const int lane = threadIdx.x & 31;
    const int64_t total = min(Q.class_chunk_base[Q.num_classes], Q.max_chunks);
    // all classes' chunks in one sequence: the counter after the classes' own
    for (int64_t j = first_chunk(Q, Q.num_classes, 0, lane); j < total;) {
        const int64_t nxt = fetch_next_chunk(Q, Q.num_classes, 0, lane);
        const Chunk ch = Q.chunks[j];
        const int t = ch.table;
        const TableDev& td = P.tables[t];
        const int64_t rows = td.rows, key_base = td.key_base;
        const int64_t k0 = ch.k0;
        const int32_t len = static_cast<int32_t>(ch.len & 0x7fffffffu);
        const int64_t bag_lo = static_cast<int64_t>(t) * P.B, bag_hi = bag_lo + P.B;
        uint32_t* keys = K.keys + k0;
        uint32_t* vals = K.vals + k0;
        BagWindow32 W = bag_window32(P, ch.first, bag_hi, k0, lane);
        for (int32_t base = 0; base < len; base += 32 * kKeygenSteps) {
            int64_t idx[kKeygenSteps];
            float wt[kKeygenSteps];
#pragma unroll
            for (int u = 0; u < kKeygenSteps; ++u) {
                const int32_t q = base + 32 * u + lane;
                idx[u] = q < len ? load_index(P.indices, k0 + q, P.is32) : 0;
                wt[u] = PACKED && P.weights && q < len ? __ldg(P.weights + k0 + q) : 1.f;
            }
#pragma unroll
            for (int u = 0; u < kKeygenSteps; ++u) {
                const int32_t q = base + 32 * u + lane;
                if (base + 32 * u >= len) break;  // warp-uniform
                const bool valid = q < len;
                int64_t my_bag;
                int32_t my_s = 0, my_e = 0;
                if (!CB_KEYGEN_MASK || !bags_by_mask(W, base + 32 * u, lane, PACKED && P.mean, my_bag, my_s, my_e))
                    find_bag32(P, W, bag_hi, k0, q, valid, lane, my_bag, my_s, my_e);
                if (!valid) continue;
                if (my_bag >= bag_hi) {  // only reachable with malformed offsets
                    set_error(P.error, CB_ERR_BAD_OFFSETS);
                    my_bag = bag_hi - 1;
                }
                // An out-of-range index takes the table's spare key (it sorts
                // after every row into a run the reduce drops) and a bag outside
                // the table: it contributes to no gradient row.
                int64_t r = idx[u];
                uint32_t bag = static_cast<uint32_t>(my_bag);
                if (r < 0 || r >= rows) {
                    set_error(P.error, CB_ERR_INDEX_OOB);
                    r = rows;
                    bag = kDeadBag;
                }
                keys[q] = static_cast<uint32_t>(key_base + r);
                if (PACKED) {
                    float c = wt[u];
                    if (P.mean && my_e > my_s) c = c / static_cast<float>(my_e - my_s);
                    vals[q] = static_cast<uint32_t>(k0 + q);
                    K.packed[k0 + q] = make_uint2(bag, __float_as_uint(c));
                } else {
                    vals[q] = bag;
                }
            }
        }
        j = __shfl_sync(kFull, nxt, 0);
    }
}

// ---------------------------------------------------------------- (3) runs

// Head flags of the kRleItems sorted keys starting at `base` (thread-blocked):
// bit i is set when key[base + i] starts a run. Full groups load as four
// 16-byte vectors; the key before the group comes from the previous lane.
__device__ __forceinline__ uint32_t head_flags(const uint32_t* keys, int64_t n, int64_t base) {
    uint32_t k[kRleItems];
    if (base + kRleItems <= n) {
        const uint4* v = reinterpret_cast<const uint4*>(keys + base);
#pragma unroll
        for (int i = 0; i < kRleItems / 4; ++i) {
            const uint4 x = __ldg(v + i);
            k[4 * i] = x.x;
            k[4 * i + 1] = x.y;
            k[4 * i + 2] = x.z;
            k[4 * i + 3] = x.w;
        }
    } else {
#pragma unroll
        for (int i = 0; i < kRleItems; ++i) k[i] = base + i < n ? __ldg(keys + base + i) : 0u;
    }
    const int lane = threadIdx.x & 31;
    uint32_t prev = __shfl_up_sync(kFull, k[kRleItems - 1], 1);
    if (lane == 0 && base > 0 && base <= n) prev = __ldg(keys + base - 1);
    uint32_t flags = 0;
#pragma unroll
    for (int i = 0; i < kRleItems; ++i) {
        const uint32_t before = i == 0 ? prev : k[i - 1];
        const bool head = base + i < n && (base + i == 0 || k[i] != before);
        flags |= head ? (1u << i) : 0u;
    }
    return flags;
}

__global__ void __launch_bounds__(kRleThreads) rle_count_kernel(const uint32_t* keys, int64_t n,
                                                                 int64_t* tile_heads) {
    __shared__ int64_t sh[33];
    const int64_t base = static_cast<int64_t>(blockIdx.x) * kRleTile + threadIdx.x * kRleItems;
    const int64_t c = __popc(head_flags(keys, n, base));
    int64_t total;
    block_excl_scan(c, sh, &total);
    if (threadIdx.x == 0) tile_heads[blockIdx.x] = total;
}

// One block over the tile counts in rounds of 1024 x 8: thread i takes 8
// consecutive counts of the round (a warp reads 2 KB contiguous), one block
// scan per round, the round's total carried into the next: 45 us on cfg5.
// (With each thread owning 1/1024 of the counts every warp load touched 32
// lines: 55 us; with 16 counts per thread, at 64 registers: 57 us.)
__global__ void __launch_bounds__(1024) rle_scan_kernel(const int64_t* tile_heads, int64_t tiles,
                                                        int64_t* tile_base, int64_t* num_unique) {
    constexpr int kPer = 8;
    __shared__ int64_t sh[33];
    int64_t carry = 0;
    for (int64_t c0 = 0; c0 < tiles; c0 += static_cast<int64_t>(blockDim.x) * kPer) {
        const int64_t i0 = c0 + static_cast<int64_t>(threadIdx.x) * kPer;
        int64_t v[kPer];
        int64_t sum = 0;
#pragma unroll
        for (int u = 0; u < kPer; ++u) {
            v[u] = i0 + u < tiles ? tile_heads[i0 + u] : 0;
            sum += v[u];
        }
        int64_t total;
        int64_t run = carry + block_excl_scan(sum, sh, &total);
#pragma unroll
        for (int u = 0; u < kPer; ++u) {
            if (i0 + u < tiles) tile_base[i0 + u] = run;
            run += v[u];
        }
        carry += total;
    }
    if (threadIdx.x == 0) *num_unique = carry;
}

#ifndef CB_RLE_FNS
#define CB_RLE_FNS 1  // find a lane's n-th head with __fns (0: clear the earlier heads one by one)
#endif

// Each warp writes its run heads (unique key, start position) 32 at a time,
// coalesced: lane l writes the warp's head x = x0 + l, found by a search over
// the lanes' head prefixes (the owning lane) and then among that lane's 16 head
// flags. With few repeats nearly every position is a head, and per-thread
// stores would land 16 apart across the warp.
__global__ void __launch_bounds__(kRleThreads) rle_write_kernel(const uint32_t* keys, int64_t n,
                                                                const int64_t* tile_base,
                                                                const int64_t* num_unique,
                                                                uint32_t* uniq, uint32_t* seg_start) {
    __shared__ int64_t sh[33];
    const int lane = threadIdx.x & 31;
    const int64_t base = static_cast<int64_t>(blockIdx.x) * kRleTile + threadIdx.x * kRleItems;
    const uint32_t flags = head_flags(keys, n, base);
    int64_t total;
    const int64_t k = block_excl_scan(__popc(flags), sh, &total);
    const int64_t wk = __shfl_sync(kFull, k, 0);                  // the warp's first head in the tile
    const int32_t mine = static_cast<int32_t>(k - wk);            // this lane's first head in the warp
    const int32_t wtot = __shfl_sync(kFull, mine + __popc(flags), 31);
    uint32_t* uo = uniq + tile_base[blockIdx.x] + wk;
    uint32_t* so = seg_start + tile_base[blockIdx.x] + wk;
    const int64_t wbase = base - static_cast<int64_t>(lane) * kRleItems;  // lane 0's first position
    for (int32_t x0 = 0; x0 < wtot; x0 += 32) {
        const int32_t x = x0 + lane;
        int j = 0;  // the last lane whose first head is at or before x: it holds head x
#pragma unroll
        for (int b = 16; b >= 1; b >>= 1)
            if (__shfl_sync(kFull, mine, j + b) <= x) j += b;
        uint32_t f = __shfl_sync(kFull, flags, j);
        const int32_t mj = __shfl_sync(kFull, mine, j);
        if (x < wtot) {
            // head x is the lane's (x - mj + 1)-th head: that set bit of its flags
            int bit;
            if (CB_RLE_FNS) {
                bit = static_cast<int>(__fns(f, 0, x - mj + 1));
            } else {
                for (int32_t r = x - mj; r > 0; --r) f &= f - 1;  // drop the lane's earlier heads
                bit = __ffs(f) - 1;
            }
            const int64_t pos = wbase + static_cast<int64_t>(j) * kRleItems + bit;
            uo[x] = __ldg(keys + pos);
            so[x] = static_cast<uint32_t>(pos);
        }
    }
    if (blockIdx.x == gridDim.x - 1 && threadIdx.x == 0) seg_start[*num_unique] = static_cast<uint32_t>(n);
}

// ---------------------------------------------------------------- (4) ranges

__global__ void __launch_bounds__(1024) bwd_finalize_kernel(Problem P, BwdOut O) {
    __shared__ int64_t sh[33];
    __shared__ int64_t run_rows, run_floats;
    const int64_t U = *O.num_unique_ws;
    // First run of each table: the first run key at or above key_base_t.
    for (int t = threadIdx.x; t <= P.T; t += blockDim.x) {
        const int64_t kb = t < P.T ? P.tables[t].key_base
                                   : P.tables[P.T - 1].key_base + P.tables[P.T - 1].rows + 1;
        int64_t a = 0, b = U;
        while (a < b) {
            const int64_t m = (a + b) >> 1;
            if (static_cast<int64_t>(O.uniq[m]) < kb) a = m + 1; else b = m;
        }
        O.table_first[t] = a;
    }
    if (threadIdx.x == 0) run_rows = run_floats = 0;
    __syncthreads();
    // A table's last run may hold its out-of-range lookups (the spare key):
    // it is not output. Output rows and floats are scanned over the rest.
    for (int t0 = 0; t0 < P.T; t0 += blockDim.x) {
        const int t = t0 + threadIdx.x;
        int64_t live = 0, dim = 0;
        if (t < P.T) {
            const TableDev& td = P.tables[t];
            const int64_t a = O.table_first[t], b = O.table_first[t + 1];
            const bool dead = b > a && static_cast<int64_t>(O.uniq[b - 1]) == td.key_base + td.rows;
            O.live_end[t] = dead ? b - 1 : b;
            live = (dead ? b - 1 : b) - a;
            dim = td.dim;
        }
        int64_t rows_total, floats_total;
        const int64_t ex_rows = block_excl_scan(live, sh, &rows_total);
        const int64_t ex_floats = block_excl_scan(live * dim, sh, &floats_total);
        if (t < P.T) {
            O.out_first[t] = run_rows + ex_rows;
            O.float_base[t] = run_floats + ex_floats;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            run_rows += rows_total;
            run_floats += floats_total;
        }
        __syncthreads();
    }
    const int64_t Uo = run_rows, F = run_floats;
    if (O.table_offsets)
        for (int t = threadIdx.x; t <= P.T; t += blockDim.x) O.table_offsets[t] = t < P.T ? O.out_first[t] : Uo;
    if (threadIdx.x == 0) {
        O.out_first[P.T] = Uo;
        O.float_base[P.T] = F;
        *O.num_unique = Uo;
        *O.num_floats = F;
        int fail = 0;
        // After a timed-out sort pass the sorted order is not trustworthy.
        if (*reinterpret_cast<volatile int*>(P.error) == CB_ERR_TIMEOUT) fail = 1;
        if (O.grads && (Uo > O.cap_rows || F > O.cap_floats)) {
            set_error(P.error, CB_ERR_CAPACITY);
            fail = 1;
        }
        *O.cap_fail = fail;
        if (O.grads && !fail) O.grad_offsets[Uo] = F;
    }
}

// ---------------------------------------------------------------- (6) fix-up

// Runs split over chunks (hot rows longer than the snap cap): each warp scans
// 32 chunks at a time for tail pieces and combines each such run in fp64. Runs
// spread over more than kHeavyPieces chunks go to a list that bwd_heavy_kernel
// combines with a whole block each.
constexpr int64_t kHeavyPieces = 32;

__device__ __forceinline__ void store_grad4(float* dst, int x0, const double (&acc)[4]) {
    *reinterpret_cast<float4*>(dst + x0) =
        make_float4(static_cast<float>(acc[0]), static_cast<float>(acc[1]),
                    static_cast<float>(acc[2]), static_cast<float>(acc[3]));
}

__global__ void __launch_bounds__(kWarpThreads) bwd_fixup_kernel(const __grid_constant__ Problem P,
                                                                 const __grid_constant__ Plan Q,
                                                                 const __grid_constant__ BwdOut O) {
    if (*O.cap_fail) return;
    const int lane = threadIdx.x & 31;
    const int64_t total = min64(Q.class_chunk_base[Q.num_classes], Q.max_chunks);
    for (int64_t base = warp_id_global() * 32; base < total; base += warps_in_grid() * 32) {
        const int64_t mine = base + lane < total ? Q.tail_owner[base + lane] : -1;
        for (uint32_t mask = __ballot_sync(kFull, mine >= 0); mask; mask &= mask - 1) {
            const int b = __ffs(mask) - 1;
            const int64_t j = base + b;
            const int64_t seg = __shfl_sync(kFull, mine, b);
            const int64_t e = O.seg_start[seg + 1];
            const int64_t m = pieces_after(Q, j, e, total);
            if (m > kHeavyPieces) {
                if (lane == 0) {
                    const uint32_t slot = atomicAdd(O.heavy_count, 1u);
                    if (slot < O.max_heavy)
                        O.heavy[slot] = make_int4(static_cast<int>(j), static_cast<int>(seg),
                                                  static_cast<int>(m), 0);
                }
                continue;
            }
            const int t = Q.chunks[j].table;
            const TableDev& td = P.tables[t];
            // A fused step takes the combined row from the chunk's tail slot.
            float* dst = O.apply ? Q.carry_tail + j * P.dmax
                                 : O.grads + O.float_base[t] + (seg - O.table_first[t]) * td.dim;
            combine_pieces(Q, j, m, td.dim, P.dmax, lane,
                           [&](int x0, double (&acc)[4]) { store_grad4(dst, x0, acc); });
        }
    }
}

// One heavy run per block: warp w adds pieces w, w + 8, ... (lanes own columns;
// fp32 groups folded into fp64), then the warps' partial sums meet in shared
// memory in warp order, after the tail piece. The order is fixed, so the result
// is deterministic.
__global__ void __launch_bounds__(kWarpThreads) bwd_heavy_kernel(const __grid_constant__ Problem P,
                                                                 const __grid_constant__ Plan Q,
                                                                 const __grid_constant__ BwdOut O) {
    __shared__ double sh[kWarpThreads / 32][512];
    if (*O.cap_fail) return;
    const uint32_t count = min64(*O.heavy_count, O.max_heavy);
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    constexpr int kWarps = kWarpThreads / 32;
    for (uint32_t h = blockIdx.x; h < count; h += gridDim.x) {
        const int4 rec = O.heavy[h];
        const int64_t j = rec.x, seg = rec.y, m = rec.z;
        const int t = Q.chunks[j].table;
        const TableDev& td = P.tables[t];
        const float* head = Q.carry_head + (j + 1) * P.dmax;
        for (int x0 = lane * 4; x0 < td.dim; x0 += 128) {
            double acc[4] = {0.0, 0.0, 0.0, 0.0};
            add_pieces(head, w, kWarps, m, P.dmax, x0, acc);
            for (int x = 0; x < 4; ++x) sh[w][x0 + x] = acc[x];
        }
        __syncthreads();
        if (w == 0) {
            float* dst = O.apply ? Q.carry_tail + j * P.dmax
                                 : O.grads + O.float_base[t] + (seg - O.table_first[t]) * td.dim;
            const float* tail = Q.carry_tail + j * P.dmax;
            for (int x0 = lane * 4; x0 < td.dim; x0 += 128) {
                const float4 a = *reinterpret_cast<const float4*>(tail + x0);
                double acc[4] = {a.x, a.y, a.z, a.w};
                for (int ww = 0; ww < kWarps; ++ww)
                    for (int x = 0; x < 4; ++x) acc[x] += sh[ww][x0 + x];
                store_grad4(dst, x0, acc);
            }
        }
        __syncthreads();
    }
}

// Fused step for the runs the fix-up combined: their full gradient row waits in
// the tail slot of the chunk where the run begins. One warp per such run.
__global__ void __launch_bounds__(kWarpThreads) bwd_apply_split_kernel(const __grid_constant__ Problem P,
                                                                       const __grid_constant__ Plan Q,
                                                                       const __grid_constant__ BwdOut O) {
    if (*O.cap_fail) return;
    const int lane = threadIdx.x & 31;
    const int64_t total = min64(Q.class_chunk_base[Q.num_classes], Q.max_chunks);
    for (int64_t base = warp_id_global() * 32; base < total; base += warps_in_grid() * 32) {
        const int64_t mine = base + lane < total ? Q.tail_owner[base + lane] : -1;
        for (uint32_t mask = __ballot_sync(kFull, mine >= 0); mask; mask &= mask - 1) {
            const int b = __ffs(mask) - 1;
            const int64_t j = base + b;
            const int64_t seg = __shfl_sync(kFull, mine, b);
            const int t = Q.chunks[j].table;
            const TableDev& td = P.tables[t];
            const int64_t row = static_cast<int64_t>(O.uniq[seg]) - td.key_base;
            const float* g = Q.carry_tail + j * P.dmax;
            float sq = 0.f;
            for (int x0 = lane * 4; x0 < td.dim; x0 += 128) {
                const float4 v = *reinterpret_cast<const float4*>(g + x0);
                sq += sq4(v);
            }
            const float scale = step_scale(O, t, row, td.dim, sq);
            for (int x0 = lane * 4; x0 < td.dim; x0 += 128)
                step_cols(td, row, x0, *reinterpret_cast<const float4*>(g + x0), scale);
        }
    }
}

// ---------------------------------------------------------------- launchers

void launch_keygen(const Problem& P, const Plan& Q, const KeyGen& K, bool packed, int64_t chunk_bound,
                   int num_sms, cudaStream_t s) {
    if (packed) {
        static int cap = occupancy_grid(keygen_kernel<true>, kWarpThreads, num_sms);
        keygen_kernel<true><<<warp_grid(chunk_bound, cap), kWarpThreads, 0, s>>>(P, Q, K);
    } else {
        static int cap = occupancy_grid(keygen_kernel<false>, kWarpThreads, num_sms);
        keygen_kernel<false><<<warp_grid(chunk_bound, cap), kWarpThreads, 0, s>>>(P, Q, K);
    }
}

int64_t rle_num_tiles(int64_t n) { return (n + kRleTile - 1) / kRleTile; }

void launch_rle(const uint32_t* keys, int64_t n, int64_t* tile_heads, int64_t* tile_base,
                int64_t* num_unique, uint32_t* uniq, uint32_t* seg_start, cudaStream_t s) {
    const int64_t tiles = rle_num_tiles(n);
    rle_count_kernel<<<static_cast<unsigned>(tiles), kRleThreads, 0, s>>>(keys, n, tile_heads);
    rle_scan_kernel<<<1, 1024, 0, s>>>(tile_heads, tiles, tile_base, num_unique);
    rle_write_kernel<<<static_cast<unsigned>(tiles), kRleThreads, 0, s>>>(keys, n, tile_base,
                                                                         num_unique, uniq, seg_start);
}

void launch_bwd_finalize(const Problem& P, const BwdOut& O, cudaStream_t s) {
    bwd_finalize_kernel<<<1, 1024, 0, s>>>(P, O);
}

void launch_bwd_reduce(const Problem& P, const Plan& Q, const BwdOut& O, const void* grad_out, int cls,
                       int vpl, int gc, bool packed, bool apply, int64_t chunk_bound, int num_sms,
                       cudaStream_t s) {
    if (P.out_dtype == CB_F16) {
        launch_bwd_reduce_f16(P, Q, O, grad_out, cls, vpl, gc, packed, apply, chunk_bound, num_sms, s);
    } else if (P.out_dtype == CB_BF16) {
        launch_bwd_reduce_bf16(P, Q, O, grad_out, cls, vpl, gc, packed, apply, chunk_bound, num_sms, s);
    } else if (apply) {
        launch_bwd_reduce_f32_apply(P, Q, O, grad_out, cls, vpl, gc, packed, chunk_bound, num_sms, s);
    } else {
        launch_bwd_reduce_f32(P, Q, O, grad_out, cls, vpl, gc, packed, chunk_bound, num_sms, s);
    }
}

void launch_bwd_fixup(const Problem& P, const Plan& Q, const BwdOut& O, int64_t chunk_bound,
                      int num_sms, cudaStream_t s) {
    cudaMemsetAsync(O.heavy_count, 0, sizeof(uint32_t), s);
    const int64_t need = (chunk_bound + kWarpThreads - 1) / kWarpThreads;  // 32 chunks per warp
    const int grid = static_cast<int>(max64(1, min64(need, static_cast<int64_t>(num_sms) * 8)));
    bwd_fixup_kernel<<<grid, kWarpThreads, 0, s>>>(P, Q, O);
    const int hgrid = static_cast<int>(max64(1, min64(O.max_heavy, static_cast<int64_t>(num_sms) * 4)));
    bwd_heavy_kernel<<<hgrid, kWarpThreads, 0, s>>>(P, Q, O);
}

void launch_bwd_apply_split(const Problem& P, const Plan& Q, const BwdOut& O, int64_t chunk_bound,
                            int num_sms, cudaStream_t s) {
    const int64_t need = (chunk_bound + kWarpThreads - 1) / kWarpThreads;  // 32 chunks per warp
    const int grid = static_cast<int>(max64(1, min64(need, static_cast<int64_t>(num_sms) * 8)));
    bwd_apply_split_kernel<<<grid, kWarpThreads, 0, s>>>(P, Q, O);
}

}  // namespace cbtbe

namespace cbtbe {

// ---------------------------------------------------------------- (7) sparse step

// The optimizer step from a row-sparse gradient already in memory (written by
// the backward). Every touched row is independent: a warp takes 32 rows, each
// lane fetches one row's id and gradient offset and finds its table by
// bisection over the per-table ranges (one round trip for all 32), then the
// warp steps the rows R at a time, issuing all their gradient, table and state
// loads before any store. Lane l owns columns 4l + 128m, m < M (the fused
// step's order, so both give the same sums of squares). Nothing is done when
// the gradient buffers were too small (the backward then wrote no rows).
#ifndef CB_APPLY_MIN_BLOCKS
#define CB_APPLY_MIN_BLOCKS 4  // resident blocks per SM for rows of up to 128 columns (wider: 2)
#endif
#ifndef CB_APPLY_ROWS_M1
#define CB_APPLY_ROWS_M1 2  // rows stepped at once for rows of up to 128 columns
#endif
constexpr int kApplyShTables = 1024;  // table offsets staged in shared memory up to this many tables

// One lane's row of a group of 32: where its stored row, gradient and state
// are, its (dim, dtype), and its previous Adagrad state.
struct ApplyRow {
    unsigned long long row;    // start of the stored row
    unsigned long long grad;   // start of its gradient
    unsigned long long state;  // its state word (Adagrad), or 0
    int shape;                 // dim << 2 | dtype (dim 0: nothing loaded or stored)
    float m0;
};

__device__ __forceinline__ ApplyRow apply_row_meta(const Problem& P, const BwdOut& O, const int64_t* toff,
                                                   int64_t u0, int64_t U, int64_t F, int lane, bool adagrad) {
    const int64_t u = min64(u0 + lane, U - 1);
    const int64_t id = __ldg(O.unique_ids + u);
    const int64_t goff = __ldg(O.grad_offsets + u);
    int lo = 0, hi = P.T;  // table_offsets[lo] <= u < table_offsets[lo + 1]
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (toff[mid] <= u) lo = mid;
        else hi = mid;
    }
    const TableDev& td = P.tables[lo];
    const int64_t row = id - td.row_base;
    // A gradient this handle's backward wrote always passes; a row that does not
    // (buffers from elsewhere) is skipped and reported, never followed outside
    // a table, the gradient or the state.
    const bool ok = row >= 0 && row < td.rows && goff >= 0 && goff + td.dim <= F;
    if (!ok && u0 + lane < U) set_error(P.error, CB_ERR_INDEX_OOB);
    ApplyRow m;
    m.row = reinterpret_cast<unsigned long long>(row_ptr(td, ok ? row : 0));
    m.grad = reinterpret_cast<unsigned long long>(O.grads + (ok ? goff : 0));
    m.state = adagrad && ok ? reinterpret_cast<unsigned long long>(O.state[lo] + row) : 0ull;
    m.shape = ((ok ? td.dim : 0) << 2) | td.dtype;
    m.m0 = m.state ? *reinterpret_cast<const float*>(m.state) : 0.f;
    return m;
}

template <int M, int R>
__global__ void __launch_bounds__(kWarpThreads, M == 1 ? CB_APPLY_MIN_BLOCKS : 2)
    apply_sparse_kernel(const __grid_constant__ Problem P, const __grid_constant__ BwdOut O) {
    static_assert(32 % R == 0, "rows per step divide the warp's 32");
    // The per-table first rows, for the bisection that finds each row's table.
    __shared__ int64_t sh_toff[kApplyShTables + 1];
    const bool staged = P.T <= kApplyShTables;
    if (staged)
        for (int t = threadIdx.x; t <= P.T; t += blockDim.x) sh_toff[t] = __ldg(O.table_offsets + t);
    __syncthreads();
    const int64_t* toff = staged ? sh_toff : O.table_offsets;
    const int lane = threadIdx.x & 31;
    const int64_t U = *O.num_unique;
    const int64_t F = *O.num_floats;
    if (U > O.cap_rows || F > O.cap_floats) return;
    const bool adagrad = O.apply == kApplyAdagrad;
    // (Loading the next group's ids, offsets and states while this group steps
    // was measured: no faster on cfg5.)
    for (int64_t u0 = warp_id_global() * 32; u0 < U; u0 += warps_in_grid() * 32) {
        const ApplyRow cur = apply_row_meta(P, O, toff, u0, U, F, lane, adagrad);
        const int rows_here = static_cast<int>(min64(32, U - u0));
        for (int r0 = 0; r0 < rows_here; r0 += R) {
            char* rp[R];
            int shape[R];
            float4 g[R][M];
            uint4 x[R][M];
#pragma unroll
            for (int i = 0; i < R; ++i) {
                rp[i] = reinterpret_cast<char*>(__shfl_sync(kFull, cur.row, r0 + i));
                const float* gp = reinterpret_cast<const float*>(__shfl_sync(kFull, cur.grad, r0 + i));
                shape[i] = __shfl_sync(kFull, cur.shape, r0 + i);
#pragma unroll
                for (int m = 0; m < M; ++m) {
                    const int x0 = lane * 4 + 128 * m;
                    if (x0 < (shape[i] >> 2)) {
                        g[i][m] = *reinterpret_cast<const float4*>(gp + x0);
                        x[i][m] = load_cols(rp[i], shape[i] & 3, x0);
                    }
                }
            }
            float scale[R];
#pragma unroll
            for (int i = 0; i < R; ++i) scale[i] = O.lr;
            if (adagrad) {
                // The Adagrad scale with the arithmetic of adagrad_scale: the R
                // rows' butterflies interleaved, then lane r0 + i, which holds
                // row r0 + i's state, takes that row's update.
                float sq[R];
#pragma unroll
                for (int i = 0; i < R; ++i) {
                    sq[i] = 0.f;
#pragma unroll
                    for (int m = 0; m < M; ++m)
                        if (lane * 4 + 128 * m < (shape[i] >> 2)) sq[i] += sq4(g[i][m]);
                }
#pragma unroll
                for (int off = 16; off >= 1; off >>= 1)
#pragma unroll
                    for (int i = 0; i < R; ++i) sq[i] += __shfl_xor_sync(kFull, sq[i], off);
                float mine = 0.f;
#pragma unroll
                for (int i = 0; i < R; ++i)
                    if (lane == r0 + i) mine = sq[i];
                float my_scale = O.lr;
                if (lane >= r0 && lane < r0 + R && lane < rows_here && cur.state) {
                    const float m = cur.m0 + mine / static_cast<float>(cur.shape >> 2);
                    *reinterpret_cast<float*>(cur.state) = m;
                    my_scale = O.lr / (sqrtf(m) + O.eps);
                }
#pragma unroll
                for (int i = 0; i < R; ++i) scale[i] = __shfl_sync(kFull, my_scale, r0 + i);
            }
#pragma unroll
            for (int i = 0; i < R; ++i) {
                if (r0 + i >= rows_here) break;  // warp-uniform
                const int dim = shape[i] >> 2;
#pragma unroll
                for (int m = 0; m < M; ++m) {
                    const int x0 = lane * 4 + 128 * m;
                    if (x0 < dim) store_step(rp[i], shape[i] & 3, x0, x[i][m], g[i][m], scale[i]);
                }
            }
        }
    }
}

template <int M, int R>
void launch_apply_sparse_m(const Problem& P, const BwdOut& O, int num_sms, cudaStream_t s) {
    static int cap = occupancy_grid(apply_sparse_kernel<M, R>, kWarpThreads, num_sms);
    apply_sparse_kernel<M, R><<<cap, kWarpThreads, 0, s>>>(P, O);
}

void launch_apply_sparse(const Problem& P, const BwdOut& O, int num_sms, cudaStream_t s) {
    if (P.dmax <= 128) launch_apply_sparse_m<1, CB_APPLY_ROWS_M1>(P, O, num_sms, s);
    else if (P.dmax <= 256) launch_apply_sparse_m<2, 4>(P, O, num_sms, s);
    else launch_apply_sparse_m<4, 2>(P, O, num_sms, s);
}

}  // namespace cbtbe
