// tbe_launch.h -- host-callable launchers of the kernels (internal to the library).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace cbtbe {

struct Problem;
struct Plan;

// One radix pass over n (key, payload) pairs, each table's range sorted on
// its own: tiles never straddle tables, digits are taken from key - key_base_t.
struct SortPass {
    const uint32_t* keys_in;
    const uint32_t* vals_in;
    uint32_t* keys_out;
    uint32_t* vals_out;
    const struct Chunk* tiles;        // table-aligned tiles of at most 4096 positions
    const int64_t* num_tiles;         // device scalar
    const int64_t* table_first_tile;  // [T + 1]
    const struct TableDev* tables;
    int64_t n;
    int shift;                   // digit = ((key - key_base_t) >> shift) & 255
    // reduce-then-scan
    const int64_t* table_pos;    // [T + 1] first position of each table
    uint32_t* tile_digits;       // [tiles][256]: digit counts, then first output slots
    uint32_t* seg_sums;          // [T][segments][256]
    int T;
    int segments;                // parts of each table's tiles in the slot scan
    // single sweep with look-back
    const uint32_t* digit_base;  // [T][stride]: this pass's 256 first output slots per table
    int base_stride;             // passes * 256
    uint32_t* status;            // [tiles * 256], zeroed before the pass
    uint32_t* tile_counter;      // zeroed before the pass
    const uint32_t* never_set;   // a zero word no kernel writes (timeout test hook)
    int force_timeout;
    int* error;
    uint64_t timeout_ns;
};

// Payload bag of a lookup whose index is out of range: outside every table's
// bags, so the reduce reads the zero row for it.
constexpr uint32_t kDeadBag = 0xffffffffu;

struct KeyGen {
    uint32_t* keys;    // [n] key_base_t + index (key_base_t + rows_t: out of range)
    uint32_t* vals;    // [n] bag id (kDeadBag when out of range), or lookup position
                       // when `packed` is used
    uint2* packed;     // [n] (bag id or kDeadBag, bits of w_i * s_b) by lookup position, or null
};

struct BwdOut {
    // workspace
    const uint32_t* seg_start;   // [U + 1]
    const uint32_t* vals_sorted; // [n]
    const uint2* packed;         // [n] or null
    const uint32_t* uniq;        // [U] sorted keys of the runs (key_base_t + r)
    int64_t* num_unique_ws;      // U, runs of out-of-range lookups included
    int64_t* table_first;        // [T + 1] first run of each table
    int64_t* live_end;           // [T] one past table t's last run of real rows
                                 // (table_first[t + 1], less the out-of-range run)
    int64_t* out_first;          // [T + 1] first output row of each table (runs of
                                 // out-of-range lookups are not output)
    int64_t* float_base;         // [T + 1]
    int* cap_fail;
    int4* heavy;                 // [max_heavy] runs left for the block-wide combine
    uint32_t* heavy_count;       // zeroed before the fix-up
    int64_t max_heavy;
    // caller's buffers
    int64_t* unique_ids;
    int64_t* table_offsets;
    int64_t* grad_offsets;
    float* grads;
    int64_t cap_rows;
    int64_t cap_floats;
    int64_t* num_unique;
    int64_t* num_floats;
    // Optimizer step fused in place of the gradient output (apply != 0): no
    // gradient buffers; every touched table row is updated where its sum ends.
    int apply;             // 0: write gradients, kApplySgd, kApplyAdagrad
    float lr;
    float eps;
    float* const* state;   // device [T] -> fp32 [rows_t] (row-wise Adagrad)
};
constexpr int kApplySgd = 1;
constexpr int kApplyAdagrad = 2;

void launch_validate_offsets(const Problem& P, int num_sms, cudaStream_t s);
// The optimizer step of O.apply from the row-sparse gradient in O's caller buffers.
void launch_apply_sparse(const Problem& P, const BwdOut& O, int num_sms, cudaStream_t s);
void launch_plan(const Problem& P, const Plan& Q, int mode, const uint32_t* seg_start,
                 const int64_t* num_unique, int num_sms, bool tables_too, cudaStream_t s);

void launch_fwd_gather(const Problem& P, const Plan& Q, void* out, int cls, int dtype, int vpl,
                       int gc, int64_t chunk_bound, int num_sms, cudaStream_t s);
void launch_fwd_fixup(const Problem& P, const Plan& Q, void* out, int64_t chunk_bound,
                      int num_sms, cudaStream_t s);

constexpr int64_t kSortTileKeys = 4096;
void launch_sort_hist(const uint32_t* keys, const struct Chunk* tiles, const int64_t* num_tiles,
                      int64_t tile_bound, const struct TableDev* tables, int passes, uint32_t* hist,
                      int num_sms, cudaStream_t s);
void launch_sort_bases(const uint32_t* hist, const int64_t* table_pos, int T, int passes,
                       uint32_t* base, cudaStream_t s);
void launch_onesweep(const SortPass& S, int64_t tile_bound, cudaStream_t s);
// Parts per table of the slot scan for a tile bound (about 16 tiles each).
int radix_segments(int64_t tile_bound, int T);
// One reduce-then-scan pass: tile counts, segment sums, slots, scatter.
void launch_radix_pass(const SortPass& S, int64_t tile_bound, cudaStream_t s);
int radix_pass_launches();  // kernels launch_radix_pass enqueues

void launch_keygen(const Problem& P, const Plan& Q, const KeyGen& K, bool packed, int64_t chunk_bound,
                   int num_sms, cudaStream_t s);
int64_t rle_num_tiles(int64_t n);
void launch_rle(const uint32_t* keys, int64_t n, int64_t* tile_heads, int64_t* tile_base,
                int64_t* num_unique, uint32_t* uniq, uint32_t* seg_start, cudaStream_t s);
void launch_bwd_finalize(const Problem& P, const BwdOut& O, cudaStream_t s);
// The segmented reduce (apply: with the optimizer step fused), dispatched on
// the grad_out type P.out_dtype; one translation unit per type.
void launch_bwd_reduce(const Problem& P, const Plan& Q, const BwdOut& O, const void* grad_out, int cls,
                       int vpl, int gc, bool packed, bool apply, int64_t chunk_bound, int num_sms,
                       cudaStream_t s);
void launch_bwd_reduce_f32(const Problem& P, const Plan& Q, const BwdOut& O, const void* grad_out, int cls,
                           int vpl, int gc, bool packed, int64_t chunk_bound, int num_sms, cudaStream_t s);
void launch_bwd_reduce_f32_apply(const Problem& P, const Plan& Q, const BwdOut& O, const void* grad_out,
                                 int cls, int vpl, int gc, bool packed, int64_t chunk_bound, int num_sms,
                                 cudaStream_t s);
void launch_bwd_reduce_f16(const Problem& P, const Plan& Q, const BwdOut& O, const void* grad_out, int cls,
                           int vpl, int gc, bool packed, bool apply, int64_t chunk_bound, int num_sms,
                           cudaStream_t s);
void launch_bwd_reduce_bf16(const Problem& P, const Plan& Q, const BwdOut& O, const void* grad_out, int cls,
                            int vpl, int gc, bool packed, bool apply, int64_t chunk_bound, int num_sms,
                            cudaStream_t s);
// Rows per warp step fixed at compile time for a row of `vecs` 16-byte vectors
// spread as (lanes, groups), or 0 when the layout is only known at run time.
inline int compile_time_groups(int vpl, int lanes, int groups) {
    if (vpl > 1) return 1;
    if (lanes * groups == 32 && (groups == 1 || groups == 2 || groups == 4 || groups == 8)) return groups;
    return 0;
}
void launch_weight_grad(const Problem& P, const Plan& Q, const void* grad_out, float* grad_w, int cls,
                        int dtype, int gc, int64_t chunk_bound, int num_sms, cudaStream_t s);
void launch_bwd_fixup(const Problem& P, const Plan& Q, const BwdOut& O, int64_t chunk_bound,
                      int num_sms, cudaStream_t s);
void launch_bwd_apply_split(const Problem& P, const Plan& Q, const BwdOut& O, int64_t chunk_bound,
                            int num_sms, cudaStream_t s);

}  // namespace cbtbe
