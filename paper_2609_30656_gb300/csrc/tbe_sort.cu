// tbe_sort.cu -- stable LSD radix sort of (row id, payload) pairs for the
// de-duplicated backward of the pooled embedding bag.
//
// One pass per 8-bit digit. The digit histograms of every pass are counted once,
// while the keys are generated; each pass then reads and writes every pair
// exactly once ("onesweep"): a block takes the next tile id from a counter,
// ranks its 4096 keys by digit (warp match + per-warp counters, stable by
// position), publishes its per-digit counts, and finds the counts of all earlier
// tiles by a decoupled look-back over their published words. The look-back wait
// is bounded in time: when it runs out the kernel records CB_ERR_TIMEOUT,
// publishes anyway so later tiles finish, and writes nothing.
#include "tbe_internal.cuh"
#include "tbe_launch.h"

namespace cbtbe {

constexpr int kSortThreads = 256;
constexpr int kSortItems = 16;
constexpr int kSortTile = kSortThreads * kSortItems;  // 4096 keys
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

__global__ void __launch_bounds__(kSortThreads, 3) onesweep_kernel(SortPass S) {
    extern __shared__ __align__(16) uint32_t sh_dyn[];
    uint32_t* sh_keys = sh_dyn;                        // tile-sorted keys
    uint32_t* sh_vals = sh_dyn + kSortTile;            // tile-sorted payloads
    uint32_t* sh_vals_in = sh_dyn + 2 * kSortTile;     // payloads in load order
    __shared__ uint32_t sh_warp[kSortWarps][kRadix];   // per-warp counts, then prefixes
    __shared__ uint32_t sh_start[kRadix];              // tile-local start of each digit
    __shared__ long long sh_goff[kRadix];              // global destination - local index
    __shared__ int64_t sh_scan[33];
    __shared__ uint32_t sh_tile;
    __shared__ int sh_abort;

    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    if (tid == 0) {
        sh_tile = atomicAdd(S.tile_counter, 1u);
        sh_abort = 0;
    }
    for (int i = tid; i < kSortWarps * kRadix; i += kSortThreads) (&sh_warp[0][0])[i] = 0;
    __syncthreads();
    const uint32_t tile = sh_tile;
    const int64_t tile_base = static_cast<int64_t>(tile) * kSortTile;
    const int tile_count = static_cast<int>(min64(kSortTile, S.n - tile_base));

    // Warp-striped load: item j of lane l is position tile_base + wid*512 + j*32 + l.
    // Payloads wait in shared memory; keys and ranks stay in registers.
    uint32_t key[kSortItems];
    uint32_t rank2[kSortItems / 2];  // two 16-bit ranks per register
#pragma unroll
    for (int j = 0; j < kSortItems; ++j) {
        const int local = wid * (32 * kSortItems) + j * 32 + lane;
        const bool valid = local < tile_count;
        key[j] = valid ? __ldg(S.keys_in + tile_base + local) : 0xffffffffu;
        if (valid) sh_vals_in[local] = __ldg(S.vals_in + tile_base + local);
    }
    const uint32_t lt_mask = (1u << lane) - 1u;
#pragma unroll
    for (int j = 0; j < kSortItems; ++j) {
        const int local = wid * (32 * kSortItems) + j * 32 + lane;
        const bool valid = local < tile_count;
        const uint32_t vmask = __ballot_sync(kFull, valid);
        const uint32_t d = (key[j] >> S.shift) & (kRadix - 1);
        uint32_t peers = 0, before = 0, r = 0;
        if (valid) {
            peers = __match_any_sync(vmask, d);
            before = sh_warp[wid][d];
            r = before + __popc(peers & lt_mask);
        }
        if (j & 1) rank2[j >> 1] |= r << 16; else rank2[j >> 1] = r;
        __syncwarp();
        if (valid && lane == __ffs(peers) - 1) sh_warp[wid][d] = before + __popc(peers);
        __syncwarp();
    }
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
    store_volatile(my_status, (tile == 0 ? kFlagIncl : kFlagAgg) | count);
    int64_t total;
    const int64_t start = block_excl_scan(count, sh_scan, &total);
    sh_start[d] = static_cast<uint32_t>(start);

    // Decoupled look-back over earlier tiles for digit d, kLookbackWindow
    // predecessors per round (independent loads), bounded in time.
    uint32_t excl = 0;
    if (tile > 0) {
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
                word[w] = kk >= 0 ? load_volatile(src) : kFlagIncl;
            }
            int used = 0;
#pragma unroll
            for (int w = 0; w < kLookbackWindow; ++w) {
                if (done || used < w) continue;      // stopped earlier in this round
                const uint32_t flag = word[w] & ~kCountMask;
                if (flag == 0) continue;             // not published yet: poll it again
                excl += word[w] & kCountMask;
                used = w + 1;
                if (flag == kFlagIncl || k - w == 0) done = true;
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
    sh_goff[d] = static_cast<long long>(S.digit_base[d]) + excl - static_cast<long long>(start);
    __syncthreads();

    // Scatter into shared memory in tile-sorted order.
#pragma unroll
    for (int j = 0; j < kSortItems; ++j) {
        const int local = wid * (32 * kSortItems) + j * 32 + lane;
        if (local < tile_count) {
            const uint32_t dd = (key[j] >> S.shift) & (kRadix - 1);
            const uint32_t r = (j & 1) ? (rank2[j >> 1] >> 16) : (rank2[j >> 1] & 0xffffu);
            const uint32_t pos = sh_start[dd] + sh_warp[wid][dd] + r;
            sh_keys[pos] = key[j];
            sh_vals[pos] = sh_vals_in[local];
        }
    }
    __syncthreads();
    if (sh_abort) return;
    // Consecutive shared slots of one digit go to consecutive global slots.
    for (int i = tid; i < tile_count; i += kSortThreads) {
        const uint32_t k2 = sh_keys[i];
        const long long dest = sh_goff[(k2 >> S.shift) & (kRadix - 1)] + i;
        if (dest >= 0 && dest < S.n) {
            S.keys_out[dest] = k2;
            S.vals_out[dest] = sh_vals[i];
        }
    }
}

// Exclusive scan of each pass's 256 digit counts (one block per pass).
__global__ void digit_scan_kernel(const uint32_t* hist, uint32_t* base) {
    __shared__ int64_t sh[33];
    const int p = blockIdx.x, d = threadIdx.x;
    int64_t total;
    const int64_t ex = block_excl_scan(hist[p * kRadix + d], sh, &total);
    base[p * kRadix + d] = static_cast<uint32_t>(ex);
}

int64_t sort_num_tiles(int64_t n) { return (n + kSortTile - 1) / kSortTile; }

void launch_digit_scan(const uint32_t* hist, uint32_t* base, int passes, cudaStream_t s) {
    digit_scan_kernel<<<passes, kRadix, 0, s>>>(hist, base);
}

constexpr int kSortDynSmem = 3 * kSortTile * sizeof(uint32_t);  // 48 KB

void launch_onesweep(const SortPass& S, cudaStream_t s) {
    static bool configured = false;
    if (!configured) {
        cudaFuncSetAttribute(onesweep_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSortDynSmem);
        configured = true;
    }
    const int64_t tiles = sort_num_tiles(S.n);
    onesweep_kernel<<<static_cast<unsigned>(tiles), kSortThreads, kSortDynSmem, s>>>(S);
}

}  // namespace cbtbe
