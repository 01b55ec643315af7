/*
 * cb_tbe.h -- C ABI of the GB300 pooled embedding-bag (table-batched embedding)
 * library: the forward lookup over jagged categorical features and its
 * de-duplicated backward.
 *
 * What the operation is, and where it comes from (Component Benchmark,
 * arXiv 2609.30656):
 *   - Abstract: recommendation models mix memory-bandwidth-bound operations
 *     with dynamic shapes from jagged categorical features;
 *   - Sec. I, Sec. III.B.1: the embedding tables are terabyte-scale and are
 *     shrunk to fit one GPU;
 *   - Sec. IV.A.2: sparse_arch performs the embedding-table lookups and is
 *     almost entirely bandwidth-bound, with low arithmetic intensity.
 * The paper gives no formula, so the operation is the standard pooled bag:
 *
 *   bag (t, b) = indices[offsets[t*B + b] .. offsets[t*B + b + 1])   (key-major)
 *   out[b, Doff_t + j] = s_b * sum_{i in bag} w_i * E_t[indices[i], j]
 *
 * with Doff_t = sum of the dims of tables before t, s_b = 1 (sum pooling) or
 * 1/L (mean pooling, L = bag length; an empty bag gives exact zeros), and
 * w_i the per-sample weight (1 without weights). A weighted mean divides by L,
 * not by the sum of the weights.
 *
 * Conventions shared by every call:
 *   - Pointers named "device" are device memory of the current CUDA device;
 *     the caller owns all of them (tables, indices, offsets, weights, outputs)
 *     and keeps them alive until the work on `stream` has finished.
 *   - All GPU work is enqueued on `stream` (0 = legacy default stream); the
 *     calls return without waiting unless CB_VALIDATE is set.
 *   - A handle is not thread-safe. Calls on one handle must be ordered on one
 *     stream, or the caller synchronises between streams.
 *   - Host-side argument errors return at once, before any GPU work.
 *     Device-side checks (index range; offsets under CB_VALIDATE) never trap:
 *     they set a sticky error word. Under CB_VALIDATE the call synchronises
 *     `stream` and returns that error; otherwise cb_tbe_get_error() returns
 *     it later. An out-of-range index (negative, or >= rows_t) contributes
 *     nothing: not to the pooled output, not to any gradient row (its row is not
 *     listed unless a valid lookup touches it) and not to any optimizer step.
 *     For mean pooling the bag length L still counts it, as in the forward.
 *   - Results are deterministic: the same inputs give bit-identical outputs.
 */
#ifndef CB_TBE_H
#define CB_TBE_H

#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    CB_OK = 0,
    CB_ERR_INVALID_ARG = 1, /* bad pointer, size, dtype, alignment or layout */
    CB_ERR_INDEX_OOB = 2,   /* an index outside [0, rows_t) (device-side)    */
    CB_ERR_BAD_OFFSETS = 3, /* offsets[0] != 0, decreasing, or last != n     */
    CB_ERR_CAPACITY = 4,    /* sparse-gradient buffers smaller than needed   */
    CB_ERR_OOM = 5,         /* workspace allocation failed                   */
    CB_ERR_CUDA = 6,        /* a CUDA runtime call failed                    */
    CB_ERR_TIMEOUT = 7      /* a bounded device-side wait gave up            */
} cb_status;

typedef enum { CB_F32 = 0, CB_F16 = 1, CB_BF16 = 2 } cb_dtype;
typedef enum { CB_POOL_SUM = 0, CB_POOL_MEAN = 1 } cb_pooling;
typedef enum { CB_I32 = 0, CB_I64 = 1 } cb_index_dtype;

/* Flags for cb_tbe_create. */
#define CB_VALIDATE 0x1u  /* check offsets on device; synchronise and return errors */
#define CB_TIMING   0x2u  /* record per-component CUDA events (cb_tbe_last_timings) */
/* Mixed precision (the paper's mixed-precision preprocessor, Sec. III): the
 * pooled output is written in fp16 / bf16 (the fp32 sums rounded to nearest
 * even), and the backward, the weight gradient and the fused optimizer step take
 * grad_out in the same type (summed in fp32; gradients stay fp32). At most one of
 * the two; every table's dim must then be a multiple of 8. Default: fp32. */
#define CB_OUT_F16  0x4u
#define CB_OUT_BF16 0x8u
/* The backward's radix passes as single sweeps with a decoupled look-back
 * (each pair read and written once per pass; a block waits, bounded in time,
 * for the counts its table's earlier tiles publish) instead of the default
 * reduce-then-scan passes (a counting read of the keys and a scan of the tile
 * counts before each scatter; no block waits on another). Same results. */
#define CB_SORT_LOOKBACK 0x200u
/* Test hook (implies CB_SORT_LOOKBACK): the first radix pass's tile 1 waits on
 * a status word that nothing writes, so its bounded wait runs out and the call
 * reports CB_ERR_TIMEOUT. */
#define CB_DEBUG_FORCE_LOOKBACK_TIMEOUT 0x100u

/* One embedding table: `rows` x `dim` values of `dtype`, row-major, at the
 * device address `data` (16-byte aligned). dim * sizeof(dtype) must be a
 * multiple of 16 bytes and dim at most 512. The library only reads it. */
typedef struct {
    const void* data;
    int64_t rows;
    int32_t dim;
    cb_dtype dtype;
} cb_table_desc;

typedef struct cb_tbe cb_tbe;

/* Creates a handle on the current CUDA device for `num_tables` tables (the
 * descriptors are copied; the table memory stays the caller's). `mode` picks
 * sum or mean pooling; `idx_dtype` is the type of both indices and offsets.
 * The sum of all rows plus num_tables must be below 2^32 (the backward's sort
 * keys: each table's rows and one spare key) and num_tables * batch below 2^31.
 * Returns CB_ERR_INVALID_ARG for a bad descriptor, CB_ERR_CUDA / CB_ERR_OOM
 * if the device set-up fails. On success *out receives the handle. */
cb_status cb_tbe_create(const cb_table_desc* tables, int32_t num_tables, cb_pooling mode,
                        cb_index_dtype idx_dtype, uint32_t flags, cb_tbe** out);

/* Grows the handle's workspace for calls up to `batch` bags per table and
 * `num_indices` lookups, so that later calls allocate nothing. Synchronises
 * the device if it has to reallocate. */
cb_status cb_tbe_reserve(cb_tbe* h, int32_t batch, int64_t num_indices);

/* Forward (the sparse_arch lookup, Sec. IV.A.2; pooled bag defined above).
 *   batch        B >= 0 bags per table
 *   indices      device [num_indices], idx_dtype; row ids within each table
 *   num_indices  n >= 0 (must equal offsets[T*B])
 *   offsets      device [T*B + 1], idx_dtype, key-major, non-decreasing, from 0
 *   per_sample_weights  device fp32 [n] or NULL
 *   out          device [B, sum of dims] of the output type (fp32; fp16 / bf16
 *                under CB_OUT_F16 / CB_OUT_BF16), row-major, 16-byte aligned;
 *                every element is written. */
cb_status cb_tbe_forward(cb_tbe* h, int32_t batch, const void* indices, int64_t num_indices,
                         const void* offsets, const float* per_sample_weights, void* out,
                         cudaStream_t stream);

/* Forward without a handle and without allocating (the paper has no
 * counterpart: this is for callers of this library that must not allocate
 * device memory, such as a plugin running inside a framework that owns all
 * device memory, or a steady-state loop where a cudaMalloc / cudaFree and the
 * device-wide synchronisation it brings are not allowed).
 * Computes exactly what cb_tbe_forward computes, with the same arguments; the
 * table descriptors are passed per call instead of through a handle.
 * Scratch comes from one fixed 16 MiB __device__ array inside this library,
 * held by every GPU that loads the library until the process exits. A call
 * needs about (n / 512 + T + 1) * (32 + 8 * max dim) bytes plus ~100 bytes per
 * table (e.g. up to ~7.9 M lookups over 100 tables of dim 128); a larger call
 * is refused with CB_ERR_CAPACITY before any GPU work.
 * The first call on each device looks up the array's device address (with
 * that device current). Every call reuses the same array (its error word is
 * cleared at the start of each call), so calls whose GPU work overlaps race:
 * do not run two at once from several threads or streams. The call checks the
 * offsets, then synchronises `stream` and reads the device-side status back
 * (as under CB_VALIDATE), which is why it cannot be called while `stream` is
 * being captured into a CUDA graph. It calls no cudaMalloc, cudaFree or
 * allocating library routine. */
cb_status cb_tbe_forward_noalloc(const cb_table_desc* tables, int32_t num_tables, cb_pooling mode,
                                 cb_index_dtype idx_dtype, int32_t batch, const void* indices,
                                 int64_t num_indices, const void* offsets,
                                 const float* per_sample_weights, float* out, cudaStream_t stream);

/* Row-sparse gradient written by cb_tbe_backward. All pointers are device
 * memory owned by the caller. U = number of distinct (table, row) pairs
 * touched by the batch; F = sum over those rows of their table's dim. */
typedef struct {
    int64_t* unique_ids;    /* [cap_rows] global ids row_base_t + row, ascending  */
    int64_t* table_offsets; /* [T + 1] first entry of each table in unique_ids    */
    int64_t* grad_offsets;  /* [cap_rows + 1] start of each row's values in grads */
    float* grads;           /* [cap_floats] packed fp32 gradient rows; NULL = only
                               count U and F (size query)                        */
    int64_t cap_rows;       /* capacity of unique_ids (>= U; n always suffices)   */
    int64_t cap_floats;     /* capacity of grads (>= F)                           */
    int64_t* num_unique;    /* device scalar: U                                   */
    int64_t* num_floats;    /* device scalar: F                                   */
} cb_sparse_grad;

/* Backward of the forward above with respect to the table rows, de-duplicated
 * per touched row (the adjoint of the pooled bag; the paper profiles training
 * steps, Sec. II and Sec. VII):
 *   G[row_base_t + r] = sum over lookups i of table t with indices[i] == r of
 *                       w_i * s_b(i) * grad_out[b(i), Doff_t : Doff_t + D_t]
 * computed by an on-device stable radix sort of (row id, lookup) pairs, a
 * run-length pass and a segmented reduction. Arguments as in cb_tbe_forward;
 * grad_out is device [B, sum of dims] of the output type (fp32 unless mixed
 * precision), 16-byte aligned; gradients are fp32. When U > cap_rows
 * or F > cap_floats nothing is written to unique_ids / grad_offsets / grads,
 * num_unique and num_floats still hold the needed sizes, and the error is
 * CB_ERR_CAPACITY (returned now under CB_VALIDATE, else by cb_tbe_get_error). */
cb_status cb_tbe_backward(cb_tbe* h, int32_t batch, const void* indices, int64_t num_indices,
                          const void* offsets, const float* per_sample_weights,
                          const void* grad_out, cb_sparse_grad* g, cudaStream_t stream);

/* Synchronises the stream of the last call, returns the sticky device-side
 * error (CB_OK if none) and clears it. */
cb_status cb_tbe_get_error(cb_tbe* h);

/* Per-component device times (ms) of the last call made with CB_TIMING, in the
 * order of cb_tbe_component_name(); synchronises on the last event. Writes at
 * most `n` entries; returns CB_ERR_INVALID_ARG without CB_TIMING. */
cb_status cb_tbe_last_timings(cb_tbe* h, float* ms, int32_t n);

/* Name of timing slot `i` ("fwd.prep", "fwd.gather", ...), NULL past the end. */
const char* cb_tbe_component_name(int32_t i);

/* Number of CUDA kernels this handle has launched since creation. */
uint64_t cb_tbe_launch_count(const cb_tbe* h);

/* Test and debugging aid (not in the paper): the order the backward's stable
 * radix sort produced. Copies, on `stream`, the sorted payloads of the last
 * cb_tbe_backward or cb_tbe_backward_apply call on this handle into the device
 * array out[num_indices]: entry k belongs to the lookup at sorted position k
 * (each table's lookups by ascending row, ties in lookup order, lookups with an
 * out-of-range index after the table's rows). The payload is the lookup's
 * position in `indices` when that call had per-sample weights or mean pooling,
 * and otherwise its bag t*B + b (0xffffffff for an out-of-range index).
 * num_indices must equal that call's; the payloads stay in the handle's
 * workspace until its next backward call or until the workspace grows.
 * CB_ERR_INVALID_ARG when no such payloads are held. */
cb_status cb_tbe_sorted_payloads(const cb_tbe* h, uint32_t* out, int64_t num_indices, cudaStream_t stream);

/* Measurement aid (not in the paper): the rate at which this GPU gathers
 * random rows out of a row set that fits in L2 (on skewed indices most rows
 * the forward gather and the backward reduce read come from L2, so this rate
 * bounds them besides the HBM bandwidth). One warp per 32 items, each lane
 * loading one 4-byte index and 16 bytes of a row per step, as those kernels
 * load, 4 steps in flight and 8 blocks of 256 threads per SM (the rate grows
 * with the warps resident); it sums what it loads and writes one sum per 32
 * items.
 *   rows         device [num_rows rows of row_bytes], 16-byte aligned, read as fp32
 *   num_rows     1 .. 2^32
 *   row_bytes    64, 128, 256 or 512
 *   indices      device uint32 [num_indices] row numbers (a number >= num_rows
 *                reads row 0)
 *   out          device fp32 [ceil(num_indices / 32)]: out[k] = the sum of every
 *                value of the rows of items 32k .. 32k + 31 (fp32, any order)
 * CB_ERR_INVALID_ARG for a bad size or pointer; CB_ERR_CUDA if the launch fails.
 * The rate is num_indices * row_bytes over the time of the call on `stream`. */
cb_status cb_gather_ceiling(const void* rows, int64_t num_rows, int32_t row_bytes, const uint32_t* indices,
                            int64_t num_indices, float* out, cudaStream_t stream);

/* The same measurement on half-precision rows with the forward's arithmetic:
 * `rows` read as fp16 and every value widened into fp32 sums by the
 * mixed-precision add (8 adds per 16 bytes, the forward gather's work per
 * stored value on fp16 tables). The rate it reaches bounds the forward gather
 * on half-precision tables served from L2. Arguments, output and errors as in
 * cb_gather_ceiling (out[k]: the fp32 sum of every fp16 value of the rows of
 * items 32k .. 32k + 31). */
cb_status cb_gather_ceiling_f16(const void* rows, int64_t num_rows, int32_t row_bytes, const uint32_t* indices,
                                int64_t num_indices, float* out, cudaStream_t stream);

/* The same measurement with the rows fetched by the tensor memory accelerator
 * (TMA): four rows per cp.async.bulk.tensor .tile::gather4 into shared memory,
 * eight gathers in flight per warp, completion signalled on an mbarrier. The
 * rows are read through a 2-D tensor map over `rows` (fp32, num_rows rows of
 * row_bytes), encoded on the host at every call. Arguments and output as in
 * cb_gather_ceiling, except:
 *   num_rows   1 .. 2^31 - 1; a row number >= num_rows reads row 0
 *   row_bytes  256 or 512
 *   error      device int, set to CB_ERR_TIMEOUT if a bounded wait on an
 *              mbarrier ran out (the kernel then stops; out is incomplete)
 * CB_ERR_CUDA when the driver's tensor-map encoder cannot be reached. */
cb_status cb_gather_ceiling_tma(const void* rows, int64_t num_rows, int32_t row_bytes, const uint32_t* indices,
                                int64_t num_indices, float* out, int* error, cudaStream_t stream);

/* Short English description of a status code. */
const char* cb_tbe_status_string(cb_status s);

/* Backward with a row-wise optimizer step fused in place of the gradient
 * output (not in the paper, which frames its benchmark as training-time but
 * names no optimizer): the de-duplicated gradient G of every touched row
 * (exactly what cb_tbe_backward computes) is applied to the table at once and
 * never written out.
 *   CB_OPT_SGD:             E[r] <- E[r] - lr * G
 *   CB_OPT_ROWWISE_ADAGRAD: m[r] <- m[r] + mean_j G[j]^2;
 *                           E[r] <- E[r] - lr * G / (sqrt(m[r]) + eps)
 * computed in fp32 and rounded once to the table's storage type (round to
 * nearest even). THIS CALL WRITES THE TABLES given to cb_tbe_create (and the
 * state arrays); each touched row is written exactly once, so the result is
 * deterministic. Untouched rows and their state are left alone.
 *   batch, indices, num_indices, offsets, per_sample_weights, grad_out: as in
 *       cb_tbe_backward
 *   kind   CB_OPT_SGD or CB_OPT_ROWWISE_ADAGRAD
 *   lr     learning rate (any finite value); eps >= 0 (Adagrad)
 *   state  Adagrad only: device array of T device pointers, state[t] -> fp32
 *          [rows_t], the running mean squared gradient of each row (start at 0);
 *          NULL for SGD
 * Errors as in cb_tbe_backward; there is no capacity error. */
typedef enum { CB_OPT_SGD = 0, CB_OPT_ROWWISE_ADAGRAD = 1 } cb_optimizer;
cb_status cb_tbe_backward_apply(cb_tbe* h, int32_t batch, const void* indices, int64_t num_indices,
                                const void* offsets, const float* per_sample_weights,
                                const void* grad_out, cb_optimizer kind, float lr, float eps,
                                float* const* state, cudaStream_t stream);

/* The same optimizer step as cb_tbe_backward_apply, applied in a second pass
 * to a row-sparse gradient that cb_tbe_backward (on this handle) has written:
 * every row of g->unique_ids[0, U) gets
 *   CB_OPT_SGD:             E[r] <- E[r] - lr * G
 *   CB_OPT_ROWWISE_ADAGRAD: m[r] <- m[r] + mean_j G[j]^2;
 *                           E[r] <- E[r] - lr * G / (sqrt(m[r]) + eps)
 * in fp32, rounded once to the storage type (round to nearest even). The
 * result is bit for bit that of cb_tbe_backward_apply on the same batch; this
 * form keeps the gradient in memory (for clipping, logging or an exchange
 * between the two passes) and overlaps the rows' loads, where the fused form
 * writes no gradient buffer.
 *   g      the buffers of a completed cb_tbe_backward (grads not NULL, 16-byte
 *          aligned); U and F are read on the device. When that call ran out of
 *          capacity (U > cap_rows or F > cap_floats) nothing is written.
 *   kind, lr, eps, state: as in cb_tbe_backward_apply
 * THIS CALL WRITES THE TABLES given to cb_tbe_create (and the state arrays).
 * Errors: CB_ERR_INVALID_ARG for a NULL or misaligned buffer, an unknown kind,
 * a NaN lr, eps < 0 or a missing state; CB_ERR_CUDA if the launch fails; a row
 * whose id or offset does not fit this handle's tables or g's F (buffers not
 * written by this handle) is skipped and sets CB_ERR_INDEX_OOB (sticky; returned
 * now under CB_VALIDATE, else by cb_tbe_get_error). */
cb_status cb_tbe_apply_sparse(cb_tbe* h, const cb_sparse_grad* g, cb_optimizer kind, float lr, float eps,
                              float* const* state, cudaStream_t stream);

/* Gradient with respect to the per-sample weights (not in the paper; the
 * pooled bag above is linear in each weight, so this is its exact derivative):
 *   grad_weights[i] = s_b * sum_j grad_out[b, Doff_t + j] * E_t[indices[i], j]
 * for lookup i of bag (t, b), s_b = 1/L (mean pooling) or 1 (sum). The weights
 * themselves are not needed. Same batch, indices, num_indices and offsets as
 * cb_tbe_forward; grad_out device [B, sum of dims] of the output type,
 * 16-byte aligned;
 * grad_weights device fp32 [num_indices], every element written (0 for an
 * out-of-range index, which also sets CB_ERR_INDEX_OOB). Deterministic. */
cb_status cb_tbe_weight_grad(cb_tbe* h, int32_t batch, const void* indices, int64_t num_indices,
                             const void* offsets, const void* grad_out, float* grad_weights,
                             cudaStream_t stream);

/* Batch-size preprocessor (Component Benchmark, Sec. III: a batch captured at a
 * small size is replicated to the production batch size, keeping the input
 * distribution). Input: a key-major batch of `batch` bags per table over
 * `num_tables` tables (indices [num_indices], offsets [T*batch + 1], optional
 * per-sample weights [num_indices]), all device memory of idx_dtype / fp32.
 * Output: factor * batch bags per table, bag r*batch + b of table t (r <
 * factor) being bag b of table t:
 *   out_indices  device [factor * num_indices]
 *   out_offsets  device [T * factor * batch + 1]
 *   out_weights  device [factor * num_indices], or NULL when the input has none
 * No handle, no allocation; invalid offsets are clamped (the output then has
 * no meaning but every access stays in bounds). CB_ERR_INVALID_ARG for null
 * buffers, factor < 1, or more than 2^31 output bags. */
cb_status cb_kjt_replicate(const void* indices, const void* offsets, const float* per_sample_weights,
                           cb_index_dtype idx_dtype, int32_t num_tables, int32_t batch,
                           int64_t num_indices, int32_t factor, void* out_indices, void* out_offsets,
                           float* out_weights, cudaStream_t stream);

/* Releases the workspace and the handle (synchronises its last stream). */
void cb_tbe_destroy(cb_tbe* h);

/* ---------------------------------------------------------------------------
 * Factorization-machine cross term on the pooled rows: the inter_arch.fm step
 * that follows the lookups in the paper's DeepFM-based model (Sec. IV.A.2,
 * bandwidth-bound element-wise and reduction passes). Each of the T fields is
 * one table's pooled row, all of one dim D: v_bt = y[b, t*D : (t+1)*D], and
 *
 *   fm[b] = sum_{t < u} <v_bt, v_bu>          (Rendle's second-order term)
 *   grad_y[b, t*D + j] = grad_fm[b] * sum_{u != t} y[b, u*D + j]
 *
 * The sums are taken in fp32 in a fixed order (deterministic). These calls
 * need no handle and allocate nothing.
 *   y           device fp32 [batch, row_stride], 16-byte aligned; field t of
 *               sample b at y + b*row_stride + t*dim (the output of
 *               cb_tbe_forward over T tables of dim D, row_stride = T*D)
 *   batch       >= 0 samples
 *   num_fields  T >= 1
 *   dim         D, a multiple of 4, 4 <= D <= 512
 *   row_stride  floats from one sample to the next, >= T*D, a multiple of 4
 * Invalid arguments return CB_ERR_INVALID_ARG before any GPU work; a failed
 * launch returns CB_ERR_CUDA. */

/* out: device fp32 [batch], fm[b]. */
cb_status cb_fm_forward(const float* y, int32_t batch, int32_t num_fields, int32_t dim,
                        int64_t row_stride, float* out, cudaStream_t stream);

/* grad_fm: device fp32 [batch]; grad_y: device fp32, the layout of y (16-byte
 * aligned); columns [0, T*D) of every row are written, the rest untouched.
 * grad_y may be passed to cb_tbe_backward as its grad_out when
 * row_stride = T*D. */
cb_status cb_fm_backward(const float* y, const float* grad_fm, int32_t batch, int32_t num_fields,
                         int32_t dim, int64_t row_stride, float* grad_y, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* CB_TBE_H */
