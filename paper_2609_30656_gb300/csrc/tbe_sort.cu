// tbe_sort.cu -- stable LSD radix sort of (row id, payload) pairs for the
// de-duplicated backward of the pooled embedding bag.
//
// A table's lookups are contiguous and its sort keys are key_base_t + r with
// r <= rows_t (r = rows_t: an out-of-range index), so each table's range is
// sorted on its own, on the bits of r only (3 passes of 8 bits for tables of
// fewer than 16M rows), in tiles of at most 4096
// positions that never straddle tables. A block ranks its tile's keys by digit
// (warp match + per-warp counters, stable by position), lays them out by digit
// in shared memory and writes each digit's run to that digit's slots of the
// output. The first output slot of each (tile, digit) is found one of two ways:
//   reduce-then-scan (default): one kernel counts every tile's digits, two
//     more scan the counts per table (segment sums, then offsets), and the
//     scatter reads its slots; no block waits on another.
//   single sweep (CB_SORT_LOOKBACK): one streaming kernel counts every pass's
//     digit histogram per table; each pass then reads and writes every pair
//     once, a block publishing its per-digit counts and finding those of the
//     table's earlier tiles by a decoupled look-back over their published
//     words. The look-back wait is bounded in time: when it runs out the kernel
//     records CB_ERR_TIMEOUT, publishes anyway so later tiles finish, and
//     writes nothing.
#include "tbe_internal.cuh"
#include "tbe_launch.h"

namespace cbtbe {

constexpr int kSortThreads = 256;
constexpr int kSortItems = 16;
constexpr int kSortTile = kSortThreads * kSortItems;  // 4096 keys
static_assert(kSortTile == kSortTileKeys, "tile size shared with the host plan");
constexpr int kRadix = 256;
constexpr int kSortWarps = kSortThreads / 32;
constexpr uint32_t kFlagAgg = 1u << 30;
constexpr uint32_t kFlagIncl = 2u << 30;
constexpr uint32_t kCountMask = (1u << 30) - 1;

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ uint32_t load_volatile(const uint32_t* p) {
    return *reinterpret_cast<const volatile uint32_t*>(p);
}
__device__ __forceinline__ void store_volatile(uint32_t* p, uint32_t v) {
    *reinterpret_cast<volatile uint32_t*>(p) = v;
}

constexpr int kLookbackWindow = 8;  // predecessor tiles inspected per look-back round

__device__ __forceinline__ uint32_t sort_digit(uint32_t key, uint32_t key_base, int shift) {
    return ((key - key_base) >> shift) & (kRadix - 1);
}

// *p += v in the lanes where `on`, returning the old value there (0 elsewhere):
// one predicated shared-memory atomic, with no branch around it.
__device__ __forceinline__ uint32_t shared_add_if(uint32_t* p, uint32_t v, bool on) {
    uint32_t old = 0;
    asm volatile(
        "{\n\t.reg .pred q;\n\tsetp.ne.u32 q, %1, 0;\n\t@q atom.shared.add.u32 %0, [%2], %3;\n\t}"
        : "+r"(old)
        : "r"(static_cast<uint32_t>(on)), "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))), "r"(v)
        : "memory");
    return old;
}

// Stable rank of a tile's keys within each warp; item j of lane l of warp w is
// tile position w*512 + j*32 + l. The lanes holding one digit in item j find
// each other (match), their lowest lane adds their number to the warp's
// counter of that digit and shares the old value. A warp's shared-memory
// atomics take effect in issue order, so item j's lanes count before item
// j + 1's, and lanes of one item by lane: the rank follows the position.
// Positions past the tile count under the extra digit kRadix. The matches of
// kRankBatch items are found before their atomics are issued (in item order),
// so that independent match, atomic and shuffle latencies overlap.
#ifndef CB_RANK_BATCH
#define CB_RANK_BATCH 2
#endif
constexpr int kRankBatch = CB_RANK_BATCH;
// NT threads per block rank a tile of kSortTile keys, NI = kSortTile / NT per thread.
template <int NT>
__device__ __forceinline__ void rank_tile(const uint32_t (&key)[kSortTile / NT], int tile_count, uint32_t key_base,
                                          int shift, uint32_t (*sh_warp)[kRadix + 1],
                                          uint32_t (&rank2)[kSortTile / NT / 2]) {
    constexpr int NI = kSortTile / NT;
    static_assert(NI % kRankBatch == 0, "rank batches divide the items");
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const uint32_t lt_mask = (1u << lane) - 1u;
#pragma unroll
    for (int j0 = 0; j0 < NI; j0 += kRankBatch) {
        uint32_t d[kRankBatch], peers[kRankBatch], before[kRankBatch];
#pragma unroll
        for (int i = 0; i < kRankBatch; ++i) {
            const int j = j0 + i;
            const int local = wid * (32 * NI) + j * 32 + lane;
            d[i] = local < tile_count ? sort_digit(key[j], key_base, shift) : kRadix;
            peers[i] = __match_any_sync(kFull, d[i]);
        }
#pragma unroll
        for (int i = 0; i < kRankBatch; ++i) {
            const int leader = __ffs(peers[i]) - 1;
            before[i] = shared_add_if(&sh_warp[wid][d[i]], static_cast<uint32_t>(__popc(peers[i])), lane == leader);
        }
#pragma unroll
        for (int i = 0; i < kRankBatch; ++i) {
            const int j = j0 + i;
            const int leader = __ffs(peers[i]) - 1;
            const uint32_t r = __shfl_sync(kFull, before[i], leader) + __popc(peers[i] & lt_mask);
            if (j & 1) rank2[j >> 1] |= r << 16; else rank2[j >> 1] = r;  // two 16-bit ranks per register
        }
    }
}

// The tile laid out by digit in shared memory (slot = the warp's start of the
// digit, which holds the digit's tile-local start plus the counts of earlier
// warps, + the rank): every slot first (the counters are read-only here), then
// the stores. With CB_SORT_KV_PAIRS each (key, payload) pair goes to shared
// memory as one 8-byte word.
#ifndef CB_SORT_KV_PAIRS
#define CB_SORT_KV_PAIRS 0
#endif
template <int NT>
__device__ __forceinline__ void scatter_tile(const uint32_t (&key)[kSortTile / NT], const uint32_t (&val)[kSortTile / NT],
                                             uint32_t (&rank2)[kSortTile / NT / 2], int tile_count, uint32_t key_base,
                                             int shift, const uint32_t (*sh_warp)[kRadix + 1],
                                             uint32_t* sh_keys, uint32_t* sh_vals) {
    constexpr int NI = kSortTile / NT;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
    for (int j = 0; j < NI; ++j) {
        const uint32_t dd = sort_digit(key[j], key_base, shift);
        const uint32_t r = (j & 1) ? (rank2[j >> 1] >> 16) : (rank2[j >> 1] & 0xffffu);
        const uint32_t pos = (sh_warp[wid][dd] + r) & 0xffffu;  // < 4096 for real items
        rank2[j >> 1] = (j & 1) ? ((rank2[j >> 1] & 0xffffu) | (pos << 16))
                                : ((rank2[j >> 1] & 0xffff0000u) | pos);
    }
#pragma unroll
    for (int j = 0; j < NI; ++j) {
        const int local = wid * (32 * NI) + j * 32 + lane;
        if (local < tile_count) {
            const uint32_t pos = (j & 1) ? (rank2[j >> 1] >> 16) : (rank2[j >> 1] & 0xffffu);
            if (CB_SORT_KV_PAIRS) {
                reinterpret_cast<uint2*>(sh_keys)[pos] = make_uint2(key[j], val[j]);
            } else {
                sh_keys[pos] = key[j];
                sh_vals[pos] = val[j];
            }
        }
    }
}

// Consecutive shared slots of one digit go to consecutive global slots
// (destination = sh_goff[digit] + slot). Half a tile at a time: its shared
// reads, its destinations, its stores.
template <int NT>
__device__ __forceinline__ void write_tile(const SortPass& S, int tile_count, uint32_t key_base,
                                           const int32_t* sh_goff, const uint32_t* sh_keys,
                                           const uint32_t* sh_vals) {
    const int tid = threadIdx.x;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        constexpr int kHalf = kSortTile / NT / 2;
        uint32_t key[kHalf], val[kHalf];
        int32_t dst[kHalf];
#pragma unroll
        for (int j = 0; j < kHalf; ++j) {
            const int i = tid + (h * kHalf + j) * NT;
            if (CB_SORT_KV_PAIRS) {
                const uint2 kv = i < tile_count ? reinterpret_cast<const uint2*>(sh_keys)[i] : make_uint2(0u, 0u);
                key[j] = kv.x;
                val[j] = kv.y;
            } else {
                key[j] = i < tile_count ? sh_keys[i] : 0u;
                val[j] = i < tile_count ? sh_vals[i] : 0u;
            }
        }
#pragma unroll
        for (int j = 0; j < kHalf; ++j)
            dst[j] = sh_goff[sort_digit(key[j], key_base, S.shift)] + tid + (h * kHalf + j) * NT;
#pragma unroll
        for (int j = 0; j < kHalf; ++j) {
            const int i = tid + (h * kHalf + j) * NT;
            if (i < tile_count && dst[j] >= 0 && dst[j] < S.n) {
                S.keys_out[dst[j]] = key[j];
                S.vals_out[dst[j]] = val[j];
            }
        }
    }
}

__global__ void __launch_bounds__(kSortThreads, 3) onesweep_kernel(SortPass S) {
    extern __shared__ __align__(16) uint32_t sh_dyn[];
    uint32_t* sh_keys = sh_dyn;                            // tile-sorted keys
    uint32_t* sh_vals = sh_dyn + kSortTile;                // tile-sorted payloads
    __shared__ uint32_t sh_warp[kSortWarps][kRadix + 1];   // per-warp counts, then prefixes
                                                           // (slot kRadix: positions past the tile)
    __shared__ int32_t sh_goff[kRadix];                    // global destination - local index
    __shared__ int64_t sh_scan[33];
    __shared__ uint32_t sh_tile;
    __shared__ int sh_abort;

    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    if (tid == 0) {
        sh_tile = atomicAdd(S.tile_counter, 1u);
        sh_abort = 0;
    }
    for (int i = tid; i < kSortWarps * (kRadix + 1); i += kSortThreads) (&sh_warp[0][0])[i] = 0;
    __syncthreads();
    const uint32_t tile = sh_tile;
    if (tile >= *S.num_tiles) return;  // the grid is an upper bound on the tiles
    const Chunk tc = S.tiles[tile];
    const int t = tc.table;
    const int64_t tile_base = tc.k0;
    const int tile_count = static_cast<int>(min64(tc.len & 0x7fffffffu, S.n - tile_base));
    const uint32_t key_base = static_cast<uint32_t>(S.tables[t].key_base);
    const int64_t first_tile = S.table_first_tile[t];

    // Warp-striped load: item j of lane l is position tile_base + wid*512 + j*32 + l.
    // Keys, payloads and ranks stay in registers until the shared scatter.
    uint32_t key[kSortItems], val[kSortItems];
#pragma unroll
    for (int j = 0; j < kSortItems; ++j) {
        const int local = wid * (32 * kSortItems) + j * 32 + lane;
        const bool valid = local < tile_count;
        key[j] = valid ? __ldg(S.keys_in + tile_base + local) : 0u;
        val[j] = valid ? __ldg(S.vals_in + tile_base + local) : 0u;
    }
    uint32_t rank2[kSortItems / 2];
    rank_tile<kSortThreads>(key, tile_count, key_base, S.shift, sh_warp, rank2);
    __syncthreads();

    // Thread d: per-warp exclusive prefix and the tile's count of digit d.
    const int d = tid;
    uint32_t count = 0;
#pragma unroll
    for (int w = 0; w < kSortWarps; ++w) {
        const uint32_t c = sh_warp[w][d];
        sh_warp[w][d] = count;
        count += c;
    }
    uint32_t* my_status = S.status + static_cast<int64_t>(tile) * kRadix + d;
    store_volatile(my_status, (tile == first_tile ? kFlagIncl : kFlagAgg) | count);
    int64_t total;
    const int64_t start = block_excl_scan(count, sh_scan, &total);
#pragma unroll
    for (int w = 0; w < kSortWarps; ++w) sh_warp[w][d] += static_cast<uint32_t>(start);

    // Decoupled look-back over earlier tiles for digit d, kLookbackWindow
    // predecessors per round (independent loads), bounded in time.
    uint32_t excl = 0;
    if (tile > first_tile) {
        int64_t k = static_cast<int64_t>(tile) - 1;
        const uint64_t t0 = global_ns();
        uint32_t spins = 0;
        bool done = false;
        while (!done) {
            uint32_t word[kLookbackWindow];
#pragma unroll
            for (int w = 0; w < kLookbackWindow; ++w) {
                const int64_t kk = k - w;
                const uint32_t* src = (S.force_timeout && tile == 1) ? S.never_set
                                                                      : S.status + kk * kRadix + d;
                word[w] = kk >= first_tile ? load_volatile(src) : kFlagIncl;
            }
            int used = 0;
#pragma unroll
            for (int w = 0; w < kLookbackWindow; ++w) {
                if (done || used < w) continue;      // stopped earlier in this round
                const uint32_t flag = word[w] & ~kCountMask;
                if (flag == 0) continue;             // not published yet: poll it again
                excl += word[w] & kCountMask;
                used = w + 1;
                if (flag == kFlagIncl || k - w <= first_tile) done = true;
            }
            k -= used;
            if (!done && used == 0) {
                // The nearest predecessor has not published yet: poll that one
                // word alone, backing off, then read the window again.
                const uint32_t* src = (S.force_timeout && tile == 1) ? S.never_set
                                                                     : S.status + k * kRadix + d;
                uint32_t ns = 32;
                bool timed_out = false;
                while ((load_volatile(src) & ~kCountMask) == 0) {
                    if ((++spins & 15u) == 0 && global_ns() - t0 > S.timeout_ns) {
                        timed_out = true;
                        break;
                    }
                    __nanosleep(ns);
                    ns = ns < 512 ? 2 * ns : ns;
                }
                if (timed_out) {
                    set_error(S.error, CB_ERR_TIMEOUT);
                    atomicExch(&sh_abort, 1);
                    break;
                }
            }
        }
        store_volatile(my_status, kFlagIncl | ((excl + count) & kCountMask));
    }
    // Positions are below 2^30 and the local index below 2^12: 32 bits suffice.
    sh_goff[d] = static_cast<int32_t>(
        static_cast<int64_t>(S.digit_base[static_cast<int64_t>(t) * S.base_stride + d]) + excl - start);
    __syncthreads();

    scatter_tile<kSortThreads>(key, val, rank2, tile_count, key_base, S.shift, sh_warp, sh_keys, sh_vals);
    __syncthreads();
    if (sh_abort) return;
    write_tile<kSortThreads>(S, tile_count, key_base, sh_goff, sh_keys, sh_vals);
}

// ---------------------------------------------------------------- reduce-then-scan

// (a) Digit counts of every tile of this pass: 16 keys per thread, shared
// counters (their order does not matter here).
#ifndef CB_COUNT_MIN_BLOCKS
#define CB_COUNT_MIN_BLOCKS 8  // resident blocks per SM the count kernel is compiled for (31 registers)
#endif
__global__ void __launch_bounds__(kSortThreads, CB_COUNT_MIN_BLOCKS) radix_count_kernel(const SortPass S) {
    __shared__ uint32_t sh[kRadix];
    const int64_t tile = blockIdx.x;
    if (tile >= *S.num_tiles) return;  // the grid is an upper bound on the tiles
    const int tid = threadIdx.x;
    sh[tid] = 0;
    const Chunk tc = S.tiles[tile];
    const int count = static_cast<int>(min64(tc.len & 0x7fffffffu, S.n - tc.k0));
    const uint32_t rb = static_cast<uint32_t>(S.tables[tc.table].key_base);
    uint32_t k[kSortItems];
#pragma unroll
    for (int j = 0; j < kSortItems; ++j) {
        const int i = tid + j * kSortThreads;
        k[j] = i < count ? __ldg(S.keys_in + tc.k0 + i) : 0u;
    }
    __syncthreads();
#pragma unroll
    for (int j = 0; j < kSortItems; ++j)
        if (tid + j * kSortThreads < count) atomicAdd(&sh[sort_digit(k[j], rb, S.shift)], 1u);
    __syncthreads();
    S.tile_digits[tile * kRadix + tid] = sh[tid];
}

// Table t's tiles [f, e) cut into S.segments equal parts; part s is [a, b).
__device__ __forceinline__ void segment_range(const SortPass& S, int t, int s, int64_t* a, int64_t* b) {
    const int64_t f = S.table_first_tile[t], e = S.table_first_tile[t + 1];
    const int64_t per = (e - f + S.segments - 1) / S.segments;
    *a = min64(f + s * per, e);
    *b = min64(*a + per, e);
}

// (b) Per (table, segment) block, thread d: the segment's count of digit d.
__global__ void __launch_bounds__(kRadix) radix_segsum_kernel(const SortPass S) {
    const int t = blockIdx.x / S.segments, sg = blockIdx.x % S.segments, d = threadIdx.x;
    int64_t a, b;
    segment_range(S, t, sg, &a, &b);
    const uint32_t* c = S.tile_digits + d;
    uint32_t sum = 0;
    int64_t k = a;
    for (; k + 8 <= b; k += 8) {
        uint32_t v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = c[(k + u) * kRadix];
#pragma unroll
        for (int u = 0; u < 8; ++u) sum += v[u];
    }
    for (; k < b; ++k) sum += c[k * kRadix];
    S.seg_sums[(static_cast<int64_t>(t) * S.segments + sg) * kRadix + d] = sum;
}

// (c) Per (table, segment) block, thread d: the first output slot of digit d in
// each of the segment's tiles, replacing its count. The slots of digit d in
// table t start at the table's first position plus the table's counts of the
// smaller digits; within the digit, tiles (and segments) keep their order.
__global__ void __launch_bounds__(kRadix) radix_offsets_kernel(const SortPass S) {
    __shared__ int64_t sh_scan[33];
    const int t = blockIdx.x / S.segments, sg = blockIdx.x % S.segments, d = threadIdx.x;
    const uint32_t* ss = S.seg_sums + static_cast<int64_t>(t) * S.segments * kRadix + d;
    uint32_t total = 0, before = 0;
    for (int q = 0; q < S.segments; ++q) {
        const uint32_t v = ss[q * kRadix];
        before += q < sg ? v : 0u;
        total += v;
    }
    int64_t all;
    const int64_t digit_start = block_excl_scan(total, sh_scan, &all);
    // positions are below 2^30: 32 bits hold every slot
    uint32_t run = static_cast<uint32_t>(S.table_pos[t] + digit_start) + before;
    int64_t a, b;
    segment_range(S, t, sg, &a, &b);
    uint32_t* c = S.tile_digits + d;
    int64_t k = a;
    for (; k + 8 <= b; k += 8) {
        uint32_t v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = c[(k + u) * kRadix];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            c[(k + u) * kRadix] = run;
            run += v[u];
        }
    }
    for (; k < b; ++k) {
        const uint32_t v = c[k * kRadix];
        c[k * kRadix] = run;
        run += v;
    }
}

// (b + c) in one kernel (CB_SORT_TABLE_SCAN): one block of 1024 threads per
// table; thread (part, d) owns digit d over a quarter of the table's tiles.
// It sums the part's counts (16 loads in flight), the block turns the four
// parts' sums into each (part, digit)'s first slot (table start + the table's
// counts of smaller digits + the earlier parts' counts of the digit), and the
// thread replaces every count of its part by the tile's first slot. No block
// waits on another; the per-(table, segment) blocks of (b) and (c) were
// latency-bound on short loops.
#ifndef CB_SORT_TABLE_SCAN
#define CB_SORT_TABLE_SCAN 1
#endif
constexpr int kScanParts = 4;
constexpr int kScanLoads = 16;

__global__ void __launch_bounds__(kRadix * kScanParts) radix_table_scan_kernel(const SortPass S) {
    __shared__ uint32_t sh_part[kScanParts][kRadix];
    __shared__ uint32_t sh_start[kRadix];
    __shared__ int64_t sh_scan[33];
    const int t = blockIdx.x;
    const int d = threadIdx.x & (kRadix - 1), part = threadIdx.x / kRadix;
    const int64_t f = S.table_first_tile[t], e = S.table_first_tile[t + 1];
    const int64_t per = (e - f + kScanParts - 1) / kScanParts;
    const int64_t a = min64(f + part * per, e), b = min64(a + per, e);
    uint32_t* c = S.tile_digits + d;
    uint32_t sum = 0;
    int64_t k = a;
    for (; k + kScanLoads <= b; k += kScanLoads) {
        uint32_t v[kScanLoads];
#pragma unroll
        for (int u = 0; u < kScanLoads; ++u) v[u] = c[(k + u) * kRadix];
#pragma unroll
        for (int u = 0; u < kScanLoads; ++u) sum += v[u];
    }
    for (; k < b; ++k) sum += c[k * kRadix];
    sh_part[part][d] = sum;
    __syncthreads();
    uint32_t total = 0, before = 0;
#pragma unroll
    for (int q = 0; q < kScanParts; ++q) {
        const uint32_t x = sh_part[q][d];
        before += q < part ? x : 0u;
        total += x;
    }
    // digit starts: the scan over the first part's threads (0..255, one per digit)
    int64_t all;
    const int64_t ex = block_excl_scan(part == 0 ? total : 0u, sh_scan, &all);
    // positions are below 2^30: 32 bits hold every slot
    if (part == 0) sh_start[d] = static_cast<uint32_t>(S.table_pos[t] + ex);
    __syncthreads();
    uint32_t run = sh_start[d] + before;
    for (k = a; k + kScanLoads <= b; k += kScanLoads) {
        uint32_t v[kScanLoads];
#pragma unroll
        for (int u = 0; u < kScanLoads; ++u) v[u] = c[(k + u) * kRadix];
#pragma unroll
        for (int u = 0; u < kScanLoads; ++u) {
            c[(k + u) * kRadix] = run;
            run += v[u];
        }
    }
    for (; k < b; ++k) {
        const uint32_t v = c[k * kRadix];
        c[k * kRadix] = run;
        run += v;
    }
}

// (d) The scatter of tile blockIdx.x: the ranking of the single-sweep kernel,
// with the first output slot of every digit read from (c). NT threads per tile
// (NT / 32 warps ranking kSortTile / NT keys per thread); threads 0..255 own one
// digit each in the prefix step.
#ifndef CB_SCATTER_THREADS
#define CB_SCATTER_THREADS 256
#endif
constexpr int kScatterThreads = CB_SCATTER_THREADS;
static_assert(kScatterThreads >= kRadix && kSortTile % kScatterThreads == 0, "scatter block shape");

template <int NT>
__global__ void __launch_bounds__(NT, NT == 256 ? 3 : 1024 / NT) radix_scatter_kernel(const SortPass S) {
    constexpr int NI = kSortTile / NT;
    constexpr int NW = NT / 32;
    extern __shared__ __align__(16) uint32_t sh_dyn[];
    uint32_t* sh_keys = sh_dyn;                            // tile-sorted keys
    uint32_t* sh_vals = sh_dyn + kSortTile;                // tile-sorted payloads
    __shared__ uint32_t sh_warp[NW][kRadix + 1];           // per-warp counts, then prefixes
                                                           // (slot kRadix: positions past the tile)
    __shared__ int32_t sh_goff[kRadix];                    // global destination - local index
    __shared__ int64_t sh_scan[33];

    const int64_t tile = blockIdx.x;
    if (tile >= *S.num_tiles) return;  // the grid is an upper bound on the tiles
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    for (int i = tid; i < NW * (kRadix + 1); i += NT) (&sh_warp[0][0])[i] = 0;
    // digit tid's first output slot
    const uint32_t slot = tid < kRadix ? S.tile_digits[tile * kRadix + tid] : 0u;
    const Chunk tc = S.tiles[tile];
    const int64_t tile_base = tc.k0;
    const int tile_count = static_cast<int>(min64(tc.len & 0x7fffffffu, S.n - tile_base));
    const uint32_t key_base = static_cast<uint32_t>(S.tables[tc.table].key_base);
    uint32_t key[NI], val[NI];
#pragma unroll
    for (int j = 0; j < NI; ++j) {
        const int local = wid * (32 * NI) + j * 32 + lane;
        const bool valid = local < tile_count;
        key[j] = valid ? __ldg(S.keys_in + tile_base + local) : 0u;
        val[j] = valid ? __ldg(S.vals_in + tile_base + local) : 0u;
    }
    __syncthreads();
    uint32_t rank2[NI / 2];
    rank_tile<NT>(key, tile_count, key_base, S.shift, sh_warp, rank2);
    __syncthreads();
    const int d = tid;
    uint32_t count = 0;
    if (d < kRadix) {
#pragma unroll
        for (int w = 0; w < NW; ++w) {
            const uint32_t c = sh_warp[w][d];
            sh_warp[w][d] = count;
            count += c;
        }
    }
    int64_t total;
    const int64_t start = block_excl_scan(count, sh_scan, &total);  // threads past 255 add 0
    if (d < kRadix) {
#pragma unroll
        for (int w = 0; w < NW; ++w) sh_warp[w][d] += static_cast<uint32_t>(start);
        sh_goff[d] = static_cast<int32_t>(static_cast<int64_t>(slot) - start);
    }
    __syncthreads();
    scatter_tile<NT>(key, val, rank2, tile_count, key_base, S.shift, sh_warp, sh_keys, sh_vals);
    __syncthreads();
    write_tile<NT>(S, tile_count, key_base, sh_goff, sh_keys, sh_vals);
}

// ---------------------------------------------------------------- single sweep

// Digit histograms of every pass, per table. Each block streams a contiguous
// range of tiles, so its shared histogram changes table only a few times.
__global__ void __launch_bounds__(256) sort_hist_kernel(const uint32_t* keys, const Chunk* tiles,
                                                        const int64_t* num_tiles,
                                                        const TableDev* tables, int passes,
                                                        uint32_t* hist) {
    __shared__ uint32_t sh[4 * kRadix];
    const int64_t nt = *num_tiles;
    const int64_t per = (nt + gridDim.x - 1) / gridDim.x;
    const int64_t lo = static_cast<int64_t>(blockIdx.x) * per, hi = min64(lo + per, nt);
    int cur = -1;
    for (int i = threadIdx.x; i < 4 * kRadix; i += blockDim.x) sh[i] = 0;
    __syncthreads();
    for (int64_t j = lo; j < hi; ++j) {
        const Chunk tc = tiles[j];
        if (tc.table != cur) {  // uniform across the block
            __syncthreads();    // every count of the previous table has landed
            if (cur >= 0) {
                for (int i = threadIdx.x; i < passes * kRadix; i += blockDim.x) {
                    if (sh[i]) atomicAdd(hist + static_cast<int64_t>(cur) * passes * kRadix + i, sh[i]);
                    sh[i] = 0;
                }
            }
            __syncthreads();    // the flush is done before new counts start
            cur = tc.table;
        }
        const uint32_t rb = static_cast<uint32_t>(tables[cur].key_base);
        const int len = static_cast<int>(tc.len & 0x7fffffffu);
        // All of the tile's loads first, then the counts.
        uint32_t r[kSortItems];
#pragma unroll
        for (int k = 0; k < kSortItems; ++k) {
            const int i = threadIdx.x + k * 256;
            r[k] = i < len ? __ldg(keys + tc.k0 + i) - rb : 0u;
        }
#pragma unroll
        for (int k = 0; k < kSortItems; ++k) {
            if (threadIdx.x + k * 256 >= len) break;
            for (int p = 0; p < passes; ++p)
                atomicAdd(&sh[p * kRadix + ((r[k] >> (8 * p)) & 255u)], 1u);
        }
    }
    __syncthreads();
    if (cur >= 0)
        for (int i = threadIdx.x; i < passes * kRadix; i += blockDim.x)
            if (sh[i]) atomicAdd(hist + static_cast<int64_t>(cur) * passes * kRadix + i, sh[i]);
}

// First output position of each digit of each pass: the table's first position
// plus the exclusive scan of that pass's digit counts (one block per table).
__global__ void sort_base_kernel(const uint32_t* hist, const int64_t* table_pos, int passes,
                                 uint32_t* base) {
    __shared__ int64_t sh[33];
    const int t = blockIdx.x, d = threadIdx.x;
    for (int p = 0; p < passes; ++p) {
        const int64_t i = (static_cast<int64_t>(t) * passes + p) * kRadix + d;
        int64_t total;
        const int64_t ex = block_excl_scan(hist[i], sh, &total);
        base[i] = static_cast<uint32_t>(table_pos[t] + ex);
    }
}

void launch_sort_hist(const uint32_t* keys, const Chunk* tiles, const int64_t* num_tiles,
                      int64_t tile_bound, const TableDev* tables, int passes, uint32_t* hist,
                      int num_sms, cudaStream_t s) {
    const int grid = static_cast<int>(max64(1, min64(tile_bound, static_cast<int64_t>(num_sms) * 4)));
    sort_hist_kernel<<<grid, 256, 0, s>>>(keys, tiles, num_tiles, tables, passes, hist);
}

void launch_sort_bases(const uint32_t* hist, const int64_t* table_pos, int T, int passes,
                       uint32_t* base, cudaStream_t s) {
    sort_base_kernel<<<T, kRadix, 0, s>>>(hist, table_pos, passes, base);
}

constexpr int kSortDynSmem = 2 * kSortTile * sizeof(uint32_t);  // 32 KB

int radix_segments(int64_t tile_bound, int T) {
    const int64_t per_table = tile_bound / max64(T, 1) + 1;
    return static_cast<int>(min64(max64((per_table + 15) / 16, 1), 1024));
}

void launch_radix_pass(const SortPass& S, int64_t tile_bound, cudaStream_t s) {
    const unsigned grid = static_cast<unsigned>(max64(tile_bound, 1));
    const unsigned parts = static_cast<unsigned>(S.T) * static_cast<unsigned>(S.segments);
    radix_count_kernel<<<grid, kSortThreads, 0, s>>>(S);
    if (CB_SORT_TABLE_SCAN) {
        radix_table_scan_kernel<<<static_cast<unsigned>(S.T), kRadix * kScanParts, 0, s>>>(S);
    } else {
        radix_segsum_kernel<<<parts, kRadix, 0, s>>>(S);
        radix_offsets_kernel<<<parts, kRadix, 0, s>>>(S);
    }
    static bool configured = false;
    if (!configured) {  // static + dynamic shared memory may pass the 48 KB default
        cudaFuncSetAttribute(radix_scatter_kernel<kScatterThreads>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kSortDynSmem);
        configured = true;
    }
    radix_scatter_kernel<kScatterThreads><<<grid, kScatterThreads, kSortDynSmem, s>>>(S);
}

int radix_pass_launches() { return CB_SORT_TABLE_SCAN ? 3 : 4; }

void launch_onesweep(const SortPass& S, int64_t tile_bound, cudaStream_t s) {
    static bool configured = false;
    if (!configured) {
        cudaFuncSetAttribute(onesweep_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSortDynSmem);
        configured = true;
    }
    onesweep_kernel<<<static_cast<unsigned>(max64(tile_bound, 1)), kSortThreads, kSortDynSmem, s>>>(S);
}

}  // namespace cbtbe
