// cb_tbe.cu -- the C ABI (include/cb_tbe.h): handle, argument checks, workspace,
// and the order of kernel launches for the forward and backward passes.
#include <algorithm>
#include <cstdint>
#include <cstring>
#include <new>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "cb_tbe.h"
#include "tbe_internal.cuh"
#include "tbe_launch.h"

using namespace cbtbe;

namespace {

#ifndef CB_FWD_CHUNK
#define CB_FWD_CHUNK 512
#endif
#ifndef CB_BWD_CHUNK
#define CB_BWD_CHUNK 512
#endif
constexpr int64_t kFwdChunk = CB_FWD_CHUNK;  // lookups per forward chunk
constexpr int64_t kBwdChunk = CB_BWD_CHUNK;  // sorted positions per reduce chunk
constexpr uint64_t kLookbackTimeoutNs = 1000000000ull;  // 1 s bounded wait
constexpr int kNumTimers = 7;
const char* const kComponentNames[kNumTimers] = {"fwd.prep",   "fwd.gather", "fwd.fixup",
                                                 "bwd.keygen", "bwd.sort",   "bwd.rle",
                                                 "bwd.reduce"};

// NVTX ranges in the shape of the component timings (the paper's hierarchical
// attribution, Sec. III.A.2): one range per entry point and, nested in it, one
// per component. They bracket the host-side launches, which a profiler then
// attributes to them; without a profiler attached they cost next to nothing.
class Ranges {
  public:
    explicit Ranges(const char* call) { nvtxRangePushA(call); }
    void phase(const char* name) {
        if (open_) nvtxRangePop();
        nvtxRangePushA(name);
        open_ = true;
    }
    ~Ranges() {
        if (open_) nvtxRangePop();
        nvtxRangePop();
    }
    Ranges(const Ranges&) = delete;
    Ranges& operator=(const Ranges&) = delete;

  private:
    bool open_ = false;
};

struct KernelClass {
    int dtype;  // storage dtype (forward) or CB_F32 (backward)
    int vpl;    // 16-byte vectors per lane: 1, 2 or 4
    int gc;     // rows per warp step fixed at compile time (0: run time)
    std::vector<int32_t> tables;
};

int elem_bytes(int dt) { return dt == CB_F32 ? 4 : 2; }

int vpl_for(int row_vecs) { return row_vecs <= 32 ? 1 : (row_vecs <= 64 ? 2 : 4); }

// Lanes per row and rows per warp step for a row of `vecs` 16-byte vectors.
void lane_split(int vecs, int32_t* lanes, int32_t* groups) {
    if (vecs >= 32) {
        *lanes = 32;
        *groups = 1;
    } else if ((vecs & (vecs - 1)) == 0) {
        *lanes = vecs;
        *groups = 32 / vecs;
    } else {
        *lanes = vecs;  // not a power of two: one row per warp step
        *groups = 1;
    }
}

size_t align_up(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

// Bump layout of the per-call workspace (pointers assigned when base != null).
struct Workspace {
    int64_t* table_pos = nullptr;
    int64_t* ord_chunk_base = nullptr;
    int64_t* class_chunk_base = nullptr;
    Chunk* chunks = nullptr;
    float* carry_head = nullptr;
    float* carry_tail = nullptr;
    int64_t* tail_owner = nullptr;
    uint32_t* chunk_next = nullptr;
    int64_t max_chunks = 0;
    // radix sort plan: table-aligned tiles
    int64_t* sp_table_pos = nullptr;
    int64_t* sp_ord = nullptr;
    int64_t* sp_class_base = nullptr;
    Chunk* sp_tiles = nullptr;
    int64_t sp_max_tiles = 0;
    // backward
    uint32_t* keys[2] = {nullptr, nullptr};
    uint32_t* vals[2] = {nullptr, nullptr};
    uint2* packed = nullptr;
    uint32_t* hist = nullptr;
    uint32_t* digit_base = nullptr;
    uint32_t* status = nullptr;
    uint32_t* tile_counters = nullptr;
    uint32_t* tile_digits = nullptr;
    uint32_t* seg_sums = nullptr;
    int segments = 1;
    int64_t* tile_heads = nullptr;
    int64_t* tile_base = nullptr;
    uint32_t* uniq = nullptr;
    uint32_t* seg_start = nullptr;
    int64_t* table_first = nullptr;
    int64_t* live_end = nullptr;
    int64_t* out_first = nullptr;
    int64_t* float_base = nullptr;
    int64_t* num_unique = nullptr;
    int64_t* out_sizes = nullptr;  // [2] U and F of a fused step (no caller buffers)
    int* cap_fail = nullptr;
    int4* heavy = nullptr;
    uint32_t* heavy_count = nullptr;
    int64_t max_heavy = 0;
    int64_t sort_tiles = 0;
    size_t status_bytes = 0;
};

}  // namespace

struct cb_tbe {
    int device = 0;
    int out_dtype = CB_F32;  // pooled output and grad_out: fp32, or fp16 / bf16 (mixed precision)
    int num_sms = 1;
    int32_t T = 0;
    int mode = CB_POOL_SUM;
    int is32 = 0;
    uint32_t flags = 0;
    int32_t sum_d = 0;
    int32_t dmax = 0;
    int64_t sum_rows = 0;
    int key_bits = 1;
    int passes = 1;
    std::vector<TableDev> tables;
    std::vector<KernelClass> fwd_classes, bwd_classes;
    // persistent device memory: tables, class lists, error word, a never-written word
    void* persist = nullptr;
    TableDev* d_tables = nullptr;
    int32_t* d_fwd_class_tables = nullptr;
    int32_t* d_fwd_class_start = nullptr;
    int32_t* d_bwd_class_tables = nullptr;
    int32_t* d_bwd_class_start = nullptr;
    int32_t* d_all_tables = nullptr;  // 0..T-1, one class: the radix sort plan
    int32_t* d_all_start = nullptr;   // {0, T}
    int* d_error = nullptr;
    uint32_t* d_never_set = nullptr;
    uint4* d_zero_row = nullptr;  // 2 KB of zeros
    // grown on demand
    void* ws = nullptr;
    size_t ws_bytes = 0;
    cudaStream_t last_stream = nullptr;
    // Sorted payloads of the last backward that reached the sort (workspace).
    const uint32_t* last_sorted = nullptr;
    int64_t last_sorted_n = 0;
    cudaEvent_t ev_fwd[4] = {};
    cudaEvent_t ev_bwd[5] = {};
    bool fwd_timed = false;
    bool bwd_timed = false;
    uint64_t launches = 0;
};

namespace {

// Computes (and, with a base, assigns) the workspace for calls up to B bags per
// table and n lookups. Returns the byte size.
size_t layout(const cb_tbe* h, int64_t B, int64_t n, char* base, Workspace* w) {
    size_t off = 0;
    auto take = [&](size_t bytes) -> void* {
        void* p = base ? static_cast<void*>(base + off) : nullptr;
        off += align_up(std::max<size_t>(bytes, 1));
        return p;
    };
    const int64_t T = h->T;
    const int64_t nc = std::max<size_t>(h->fwd_classes.size(), h->bwd_classes.size());
    const int64_t chunk = std::min(kFwdChunk, kBwdChunk);
    const int64_t max_chunks = n / chunk + T + 1;
    Workspace ws;
    ws.max_chunks = max_chunks;
    ws.table_pos = static_cast<int64_t*>(take(sizeof(int64_t) * (T + 1)));
    ws.ord_chunk_base = static_cast<int64_t*>(take(sizeof(int64_t) * (T + 1)));
    ws.class_chunk_base = static_cast<int64_t*>(take(sizeof(int64_t) * (nc + 1)));
    ws.chunks = static_cast<Chunk*>(take(sizeof(Chunk) * max_chunks));
    ws.carry_head = static_cast<float*>(take(sizeof(float) * max_chunks * h->dmax));
    ws.carry_tail = static_cast<float*>(take(sizeof(float) * max_chunks * h->dmax));
    ws.tail_owner = static_cast<int64_t*>(take(sizeof(int64_t) * max_chunks));
    ws.chunk_next = static_cast<uint32_t*>(take(sizeof(uint32_t) * (nc + 1)));
    for (int i = 0; i < 2; ++i) {
        ws.keys[i] = static_cast<uint32_t*>(take(sizeof(uint32_t) * n));
        ws.vals[i] = static_cast<uint32_t*>(take(sizeof(uint32_t) * n));
    }
    ws.packed = static_cast<uint2*>(take(sizeof(uint2) * n));
    ws.sp_max_tiles = n / kSortTileKeys + T + 1;
    ws.sp_table_pos = static_cast<int64_t*>(take(sizeof(int64_t) * (T + 1)));
    ws.sp_ord = static_cast<int64_t*>(take(sizeof(int64_t) * (T + 1)));
    ws.sp_class_base = static_cast<int64_t*>(take(sizeof(int64_t) * 2));
    ws.sp_tiles = static_cast<Chunk*>(take(sizeof(Chunk) * ws.sp_max_tiles));
    ws.sort_tiles = ws.sp_max_tiles;
    if (h->flags & (CB_SORT_LOOKBACK | CB_DEBUG_FORCE_LOOKBACK_TIMEOUT)) {
        const size_t hist_words = static_cast<size_t>(T) * h->passes * 256;
        ws.digit_base = static_cast<uint32_t*>(take(sizeof(uint32_t) * hist_words));
        ws.status_bytes = sizeof(uint32_t) * static_cast<size_t>(h->passes) * ws.sort_tiles * 256;
        // histograms, status words and tile counters are adjacent: one memset clears them
        ws.hist = static_cast<uint32_t*>(take(sizeof(uint32_t) * hist_words + ws.status_bytes +
                                              sizeof(uint32_t) * 4));
        ws.status = base ? ws.hist + hist_words : nullptr;
        ws.tile_counters = base ? ws.status + static_cast<size_t>(h->passes) * ws.sort_tiles * 256 : nullptr;
        ws.status_bytes += sizeof(uint32_t) * hist_words + sizeof(uint32_t) * 4;  // cleared from `hist` on
    } else {
        ws.segments = radix_segments(ws.sp_max_tiles, static_cast<int>(T));
        ws.tile_digits = static_cast<uint32_t*>(take(sizeof(uint32_t) * 256 * ws.sort_tiles));
        ws.seg_sums = static_cast<uint32_t*>(take(sizeof(uint32_t) * 256 * T * ws.segments));
    }
    const int64_t rt = rle_num_tiles(n);
    ws.tile_heads = static_cast<int64_t*>(take(sizeof(int64_t) * rt));
    ws.tile_base = static_cast<int64_t*>(take(sizeof(int64_t) * rt));
    ws.uniq = static_cast<uint32_t*>(take(sizeof(uint32_t) * n));
    ws.seg_start = static_cast<uint32_t*>(take(sizeof(uint32_t) * (n + 1)));
    ws.table_first = static_cast<int64_t*>(take(sizeof(int64_t) * (T + 1)));
    ws.live_end = static_cast<int64_t*>(take(sizeof(int64_t) * T));
    ws.out_first = static_cast<int64_t*>(take(sizeof(int64_t) * (T + 1)));
    ws.float_base = static_cast<int64_t*>(take(sizeof(int64_t) * (T + 1)));
    ws.num_unique = static_cast<int64_t*>(take(sizeof(int64_t)));
    ws.out_sizes = static_cast<int64_t*>(take(sizeof(int64_t) * 2));
    ws.cap_fail = static_cast<int*>(take(sizeof(int)));
    ws.max_heavy = max_chunks / 32 + 1;  // a heavy run owns more than 32 chunks
    ws.heavy = static_cast<int4*>(take(sizeof(int4) * ws.max_heavy));
    ws.heavy_count = static_cast<uint32_t*>(take(sizeof(uint32_t)));
    if (w) *w = ws;
    return off;
}

cb_status ensure_workspace(cb_tbe* h, int64_t B, int64_t n) {
    const size_t need = layout(h, B, n, nullptr, nullptr);
    if (need <= h->ws_bytes) return CB_OK;
    if (h->ws) {
        cudaDeviceSynchronize();
        cudaFree(h->ws);
        h->ws = nullptr;
        h->ws_bytes = 0;
        h->last_sorted = nullptr;
    }
    if (cudaMalloc(&h->ws, need) != cudaSuccess) {
        cudaGetLastError();
        h->ws = nullptr;
        return CB_ERR_OOM;
    }
    h->ws_bytes = need;
    return CB_OK;
}

bool current_device_ok(const cb_tbe* h) {
    int dev = -1;
    return cudaGetDevice(&dev) == cudaSuccess && dev == h->device;
}

Problem make_problem(const cb_tbe* h, int32_t B, const void* indices, int64_t n, const void* offsets,
                     const float* weights) {
    Problem P;
    P.tables = h->d_tables;
    P.zero_row = h->d_zero_row;
    P.indices = indices;
    P.offsets = offsets;
    P.weights = weights;
    P.error = h->d_error;
    P.n = n;
    P.T = h->T;
    P.B = B;
    P.sum_d = h->sum_d;
    P.is32 = h->is32;
    P.mean = h->mode == CB_POOL_MEAN;
    P.dmax = h->dmax;
    P.out_dtype = h->out_dtype;
    return P;
}

Plan make_plan(const cb_tbe* h, const Workspace& w, bool bwd, int64_t chunk_len) {
    Plan Q;
    Q.chunk_len = static_cast<int32_t>(chunk_len);
    // Chunk boundaries move to the end of the bag / run they cut unless it is
    // longer than this, so only heavy bags and hot rows are split.
    Q.snap_cap = static_cast<int32_t>(bwd ? chunk_len : 4 * chunk_len);
    Q.num_classes = static_cast<int32_t>(bwd ? h->bwd_classes.size() : h->fwd_classes.size());
    Q.class_tables = bwd ? h->d_bwd_class_tables : h->d_fwd_class_tables;
    Q.class_table_start = bwd ? h->d_bwd_class_start : h->d_fwd_class_start;
    Q.table_pos = w.table_pos;
    Q.ord_chunk_base = w.ord_chunk_base;
    Q.class_chunk_base = w.class_chunk_base;
    Q.chunks = w.chunks;
    Q.max_chunks = w.max_chunks;
    Q.carry_head = w.carry_head;
    Q.carry_tail = w.carry_tail;
    Q.tail_owner = w.tail_owner;
    Q.chunk_next = w.chunk_next;
    return Q;
}

cb_status finish_call(cb_tbe* h, cudaStream_t stream) {
    if (cudaGetLastError() != cudaSuccess) return CB_ERR_CUDA;
    h->last_stream = stream;
    if (h->flags & CB_VALIDATE) return cb_tbe_get_error(h);
    return CB_OK;
}

void record(cb_tbe* h, cudaEvent_t e, cudaStream_t s) {
    if (h->flags & CB_TIMING) cudaEventRecord(e, s);
}

cb_status check_common(const cb_tbe* h, int32_t batch, const void* indices, int64_t n,
                       const void* offsets) {
    if (!h || batch < 0 || n < 0 || !offsets || (n > 0 && !indices)) return CB_ERR_INVALID_ARG;
    if (static_cast<int64_t>(h->T) * batch >= (int64_t(1) << 31)) return CB_ERR_INVALID_ARG;
    return CB_OK;
}

bool optimizer_ok(cb_optimizer kind, float lr, float eps, float* const* state) {
    if (kind != CB_OPT_SGD && kind != CB_OPT_ROWWISE_ADAGRAD) return false;
    return lr == lr && eps >= 0.f && (kind == CB_OPT_SGD || state);
}

struct ApplyArgs {
    int kind;
    float lr;
    float eps;
    float* const* state;
};

// The backward: into the caller's sparse-gradient buffers (g), or, with an
// optimizer step (a), into the tables themselves.
cb_status backward_impl(cb_tbe* h, int32_t batch, const void* indices, int64_t num_indices,
                        const void* offsets, const float* per_sample_weights, const void* grad_out,
                        cb_sparse_grad* g, const ApplyArgs* a, cudaStream_t stream) {
    cb_status st = check_common(h, batch, indices, num_indices, offsets);
    if (st != CB_OK) return st;
    const int64_t n = num_indices;
    if (n >= (int64_t(1) << 30)) return CB_ERR_INVALID_ARG;
    if (n > 0 && batch > 0 && (!grad_out || (reinterpret_cast<uintptr_t>(grad_out) & 15u)))
        return CB_ERR_INVALID_ARG;
    if (!current_device_ok(h)) return CB_ERR_INVALID_ARG;
    h->last_stream = stream;
    h->bwd_timed = false;
    h->last_sorted = nullptr;
    Problem P = make_problem(h, batch, indices, n, offsets, per_sample_weights);
    Ranges nv(a ? "cb_tbe_backward_apply" : "cb_tbe_backward");
    nv.phase("bwd.keygen");
    record(h, h->ev_bwd[0], stream);
    if ((h->flags & CB_VALIDATE) && batch > 0) {
        launch_validate_offsets(P, h->num_sms, stream);
        h->launches += 1;
    }
    if ((n == 0 || batch == 0) && a) return finish_call(h, stream);  // no row is touched
    if (n == 0 || batch == 0) {
        bool ok = cudaMemsetAsync(g->table_offsets, 0, sizeof(int64_t) * (h->T + 1), stream) == cudaSuccess;
        ok = ok && cudaMemsetAsync(g->num_unique, 0, sizeof(int64_t), stream) == cudaSuccess;
        ok = ok && cudaMemsetAsync(g->num_floats, 0, sizeof(int64_t), stream) == cudaSuccess;
        if (g->grads) ok = ok && cudaMemsetAsync(g->grad_offsets, 0, sizeof(int64_t), stream) == cudaSuccess;
        if (!ok) return CB_ERR_CUDA;
        return finish_call(h, stream);
    }
    st = ensure_workspace(h, batch, n);
    if (st != CB_OK) return st;
    Workspace w;
    layout(h, batch, n, static_cast<char*>(h->ws), &w);
    Plan Q = make_plan(h, w, true, kBwdChunk);
    const int64_t bound = n / kBwdChunk + h->T + 1;
    const bool packed = per_sample_weights != nullptr || h->mode == CB_POOL_MEAN;

    // (1) keys and payloads
    launch_plan(P, Q, 0, nullptr, nullptr, h->num_sms, true, stream);
    h->launches += 2;
    const bool lookback = (h->flags & (CB_SORT_LOOKBACK | CB_DEBUG_FORCE_LOOKBACK_TIMEOUT)) != 0;
    if (lookback && cudaMemsetAsync(w.hist, 0, w.status_bytes, stream) != cudaSuccess) return CB_ERR_CUDA;
    KeyGen K;
    K.keys = w.keys[0];
    K.vals = w.vals[0];
    K.packed = packed ? w.packed : nullptr;
    launch_keygen(P, Q, K, packed, bound, h->num_sms, stream);
    h->launches += 1;
    record(h, h->ev_bwd[1], stream);
    nv.phase("bwd.sort");

    // (2) radix sort of each table's range, 8 bits of the row number per pass
    Plan SQ;
    SQ.chunk_len = static_cast<int32_t>(kSortTileKeys);
    SQ.snap_cap = 0;
    SQ.num_classes = 1;
    SQ.class_tables = h->d_all_tables;
    SQ.class_table_start = h->d_all_start;
    SQ.table_pos = w.sp_table_pos;
    SQ.ord_chunk_base = w.sp_ord;
    SQ.class_chunk_base = w.sp_class_base;
    SQ.chunks = w.sp_tiles;
    SQ.max_chunks = w.sp_max_tiles;
    SQ.carry_head = SQ.carry_tail = nullptr;
    SQ.tail_owner = nullptr;
    SQ.chunk_next = nullptr;
    launch_plan(P, SQ, 2, nullptr, nullptr, h->num_sms, true, stream);
    h->launches += 2;
    if (lookback) {
        launch_sort_hist(w.keys[0], w.sp_tiles, w.sp_class_base + 1, w.sp_max_tiles, h->d_tables,
                         h->passes, w.hist, h->num_sms, stream);
        launch_sort_bases(w.hist, w.sp_table_pos, h->T, h->passes, w.digit_base, stream);
        h->launches += 2;
    }
    int cur = 0;
    for (int p = 0; p < h->passes; ++p) {
        SortPass S{};
        S.keys_in = w.keys[cur];
        S.vals_in = w.vals[cur];
        S.keys_out = w.keys[cur ^ 1];
        S.vals_out = w.vals[cur ^ 1];
        S.tiles = w.sp_tiles;
        S.num_tiles = w.sp_class_base + 1;
        S.table_first_tile = w.sp_ord;
        S.tables = h->d_tables;
        S.n = n;
        S.shift = 8 * p;
        if (lookback) {
            S.digit_base = w.digit_base + 256 * p;
            S.base_stride = 256 * h->passes;
            S.status = w.status + static_cast<size_t>(p) * w.sort_tiles * 256;
            S.tile_counter = w.tile_counters + p;
            S.never_set = h->d_never_set;
            S.force_timeout = (h->flags & CB_DEBUG_FORCE_LOOKBACK_TIMEOUT) && p == 0;
            S.error = h->d_error;
            S.timeout_ns = kLookbackTimeoutNs;
            launch_onesweep(S, w.sp_max_tiles, stream);
            h->launches += 1;
        } else {
            S.table_pos = w.sp_table_pos;
            S.tile_digits = w.tile_digits;
            S.seg_sums = w.seg_sums;
            S.T = h->T;
            S.segments = w.segments;
            launch_radix_pass(S, w.sp_max_tiles, stream);
            h->launches += radix_pass_launches();
        }
        cur ^= 1;
    }
    record(h, h->ev_bwd[2], stream);
    nv.phase("bwd.rle");
    h->last_sorted = w.vals[cur];
    h->last_sorted_n = n;

    // (3) runs of equal ids, (4) per-table ranges and capacity check
    launch_rle(w.keys[cur], n, w.tile_heads, w.tile_base, w.num_unique, w.uniq, w.seg_start, stream);
    h->launches += 3;
    BwdOut O;
    O.seg_start = w.seg_start;
    O.vals_sorted = w.vals[cur];
    O.packed = packed ? w.packed : nullptr;
    O.uniq = w.uniq;
    O.num_unique_ws = w.num_unique;
    O.table_first = w.table_first;
    O.live_end = w.live_end;
    O.out_first = w.out_first;
    O.float_base = w.float_base;
    O.cap_fail = w.cap_fail;
    O.heavy = w.heavy;
    O.heavy_count = w.heavy_count;
    O.max_heavy = w.max_heavy;
    if (a) {
        // No caller buffers: the sizes land in the workspace's own words.
        O.unique_ids = nullptr;
        O.table_offsets = nullptr;
        O.grad_offsets = nullptr;
        O.grads = nullptr;
        O.cap_rows = O.cap_floats = INT64_MAX;
        O.num_unique = w.out_sizes;
        O.num_floats = w.out_sizes + 1;
        O.apply = a->kind;
        O.lr = a->lr;
        O.eps = a->eps;
        O.state = a->state;
    } else {
        O.unique_ids = g->unique_ids;
        O.table_offsets = g->table_offsets;
        O.grad_offsets = g->grad_offsets;
        O.grads = g->grads;
        O.cap_rows = g->cap_rows;
        O.cap_floats = g->cap_floats;
        O.num_unique = g->num_unique;
        O.num_floats = g->num_floats;
        O.apply = 0;
        O.lr = O.eps = 0.f;
        O.state = nullptr;
    }
    const bool reduce = a || g->grads;  // a sizing call stops after the run counts
    launch_bwd_finalize(P, O, stream);
    h->launches += 1;
    if (reduce) launch_plan(P, Q, 1, w.seg_start, w.num_unique, h->num_sms, false, stream);
    if (reduce) h->launches += 1;
    record(h, h->ev_bwd[3], stream);
    nv.phase("bwd.reduce");

    // (5) segmented reduce, (6) fix-up of runs split across chunks
    if (reduce) {
        for (size_t c = 0; c < h->bwd_classes.size(); ++c) {
            launch_bwd_reduce(P, Q, O, grad_out, static_cast<int>(c), h->bwd_classes[c].vpl, h->bwd_classes[c].gc,
                              packed, a != nullptr, bound, h->num_sms, stream);
            h->launches += 1;
        }
        launch_bwd_fixup(P, Q, O, bound, h->num_sms, stream);
        h->launches += 2;
        if (a) {
            launch_bwd_apply_split(P, Q, O, bound, h->num_sms, stream);
            h->launches += 1;
        }
    }
    record(h, h->ev_bwd[4], stream);
    h->bwd_timed = (h->flags & CB_TIMING) != 0;
    return finish_call(h, stream);
}

}  // namespace

extern "C" {

const char* cb_tbe_status_string(cb_status s) {
    switch (s) {
        case CB_OK: return "ok";
        case CB_ERR_INVALID_ARG: return "invalid argument";
        case CB_ERR_INDEX_OOB: return "index out of range";
        case CB_ERR_BAD_OFFSETS: return "malformed offsets";
        case CB_ERR_CAPACITY: return "sparse-gradient capacity too small";
        case CB_ERR_OOM: return "out of device memory";
        case CB_ERR_CUDA: return "CUDA runtime error";
        case CB_ERR_TIMEOUT: return "bounded device wait timed out";
    }
    return "unknown status";
}

const char* cb_tbe_component_name(int32_t i) {
    return (i >= 0 && i < kNumTimers) ? kComponentNames[i] : nullptr;
}

cb_status cb_tbe_create(const cb_table_desc* tables, int32_t num_tables, cb_pooling mode,
                        cb_index_dtype idx_dtype, uint32_t flags, cb_tbe** out) {
    if (!out || !tables || num_tables <= 0) return CB_ERR_INVALID_ARG;
    *out = nullptr;
    if (mode != CB_POOL_SUM && mode != CB_POOL_MEAN) return CB_ERR_INVALID_ARG;
    if (idx_dtype != CB_I32 && idx_dtype != CB_I64) return CB_ERR_INVALID_ARG;
    auto* h = new (std::nothrow) cb_tbe();
    if (!h) return CB_ERR_OOM;
    h->T = num_tables;
    h->mode = mode;
    h->is32 = idx_dtype == CB_I32;
    h->flags = flags;
    if ((flags & CB_OUT_F16) && (flags & CB_OUT_BF16)) {
        delete h;
        return CB_ERR_INVALID_ARG;
    }
    h->out_dtype = (flags & CB_OUT_F16) ? CB_F16 : ((flags & CB_OUT_BF16) ? CB_BF16 : CB_F32);
    const int out_eb = elem_bytes(h->out_dtype);
    int64_t row_base = 0, doff = 0;
    for (int32_t t = 0; t < num_tables; ++t) {
        const cb_table_desc& d = tables[t];
        const bool dt_ok = d.dtype == CB_F32 || d.dtype == CB_F16 || d.dtype == CB_BF16;
        if (!dt_ok || d.rows < 0 || d.dim <= 0 || (d.rows > 0 && !d.data) ||
            (reinterpret_cast<uintptr_t>(d.data) & 15u)) {
            delete h;
            return CB_ERR_INVALID_ARG;
        }
        const int64_t row_bytes = static_cast<int64_t>(d.dim) * elem_bytes(d.dtype);
        // grad_out rows of each table (the output's type) are whole 16-byte vectors too
        if (row_bytes % 16 != 0 || row_bytes > 2048 || (static_cast<int64_t>(d.dim) * out_eb) % 16 != 0) {
            delete h;
            return CB_ERR_INVALID_ARG;
        }
        TableDev td{};
        td.data = d.data;
        td.rows = d.rows;
        td.row_base = row_base;
        td.key_base = row_base + t;  // one spare key per table: out-of-range lookups
        td.dim = d.dim;
        td.doff = static_cast<int32_t>(doff);
        td.dtype = d.dtype;
        td.row_vecs = static_cast<int32_t>(row_bytes / 16);
        lane_split(td.row_vecs, &td.lanes, &td.groups);
        td.grad_vecs = d.dim * out_eb / 16;  // grad_out row, in the output's type
        lane_split(td.grad_vecs, &td.grad_lanes, &td.grad_groups);
        row_base += d.rows;
        doff += d.dim;
        h->dmax = std::max(h->dmax, d.dim);
        h->tables.push_back(td);
    }
    // Backward keys: every table's rows plus one spare key, all below 2^32.
    if (row_base + num_tables >= (int64_t(1) << 32) || doff >= (int64_t(1) << 31) || h->dmax > 512) {
        delete h;
        return CB_ERR_INVALID_ARG;
    }
    h->sum_rows = row_base;
    h->sum_d = static_cast<int32_t>(doff);
    // Each table's range is sorted on its own, on the bits of the row number
    // r <= rows_t (r = rows_t: an out-of-range lookup).
    int64_t max_rows = 1;
    for (const TableDev& td : h->tables) max_rows = std::max(max_rows, td.rows);
    int bits = 1;
    while (bits < 32 && (int64_t(1) << bits) <= max_rows) ++bits;
    h->key_bits = bits;
    h->passes = (bits + 7) / 8;

    // Kernel classes: forward by (storage dtype, vectors per lane), backward by
    // vectors per lane of the grad_out row (fp32, or the mixed-precision type).
    for (int32_t t = 0; t < num_tables; ++t) {
        TableDev& td = h->tables[t];
        const int fv = vpl_for(td.row_vecs), bv = vpl_for(td.grad_vecs);
        const int fg = compile_time_groups(fv, td.lanes, td.groups);
        const int bg = compile_time_groups(bv, td.grad_lanes, td.grad_groups);
        auto put = [&](std::vector<KernelClass>& cls, int dt, int v, int gc) {
            for (size_t c = 0; c < cls.size(); ++c)
                if (cls[c].dtype == dt && cls[c].vpl == v && cls[c].gc == gc) {
                    cls[c].tables.push_back(t);
                    return static_cast<int>(c);
                }
            cls.push_back({dt, v, gc, {t}});
            return static_cast<int>(cls.size() - 1);
        };
        td.fwd_class = put(h->fwd_classes, td.dtype, fv, fg);
        td.bwd_class = put(h->bwd_classes, h->out_dtype, bv, bg);
    }

    if (cudaGetDevice(&h->device) != cudaSuccess ||
        cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device) != cudaSuccess) {
        cudaGetLastError();
        delete h;
        return CB_ERR_CUDA;
    }
    // Persistent block: tables | fwd class tables | fwd starts | bwd class tables | bwd starts | error | never-set
    std::vector<int32_t> fct, fcs{0}, bct, bcs{0};
    for (auto& c : h->fwd_classes) {
        fct.insert(fct.end(), c.tables.begin(), c.tables.end());
        fcs.push_back(static_cast<int32_t>(fct.size()));
    }
    for (auto& c : h->bwd_classes) {
        bct.insert(bct.end(), c.tables.begin(), c.tables.end());
        bcs.push_back(static_cast<int32_t>(bct.size()));
    }
    size_t off = 0;
    const size_t o_tab = off; off += align_up(sizeof(TableDev) * num_tables);
    const size_t o_fct = off; off += align_up(sizeof(int32_t) * fct.size());
    const size_t o_fcs = off; off += align_up(sizeof(int32_t) * fcs.size());
    const size_t o_bct = off; off += align_up(sizeof(int32_t) * bct.size());
    const size_t o_bcs = off; off += align_up(sizeof(int32_t) * bcs.size());
    std::vector<int32_t> all(num_tables), all_start{0, num_tables};
    for (int32_t t = 0; t < num_tables; ++t) all[t] = t;
    const size_t o_all = off; off += align_up(sizeof(int32_t) * num_tables);
    const size_t o_alls = off; off += align_up(sizeof(int32_t) * 2);
    const size_t o_err = off; off += align_up(sizeof(int) + sizeof(uint32_t));
    const size_t o_zero = off; off += align_up(2048);
    if (cudaMalloc(&h->persist, off) != cudaSuccess) {
        cudaGetLastError();
        delete h;
        return CB_ERR_OOM;
    }
    char* p = static_cast<char*>(h->persist);
    h->d_tables = reinterpret_cast<TableDev*>(p + o_tab);
    h->d_fwd_class_tables = reinterpret_cast<int32_t*>(p + o_fct);
    h->d_fwd_class_start = reinterpret_cast<int32_t*>(p + o_fcs);
    h->d_bwd_class_tables = reinterpret_cast<int32_t*>(p + o_bct);
    h->d_bwd_class_start = reinterpret_cast<int32_t*>(p + o_bcs);
    h->d_all_tables = reinterpret_cast<int32_t*>(p + o_all);
    h->d_all_start = reinterpret_cast<int32_t*>(p + o_alls);
    h->d_error = reinterpret_cast<int*>(p + o_err);
    h->d_never_set = reinterpret_cast<uint32_t*>(p + o_err + sizeof(int));
    h->d_zero_row = reinterpret_cast<uint4*>(p + o_zero);
    bool ok = cudaMemcpy(h->d_tables, h->tables.data(), sizeof(TableDev) * num_tables,
                         cudaMemcpyHostToDevice) == cudaSuccess;
    ok = ok && cudaMemcpy(h->d_fwd_class_tables, fct.data(), sizeof(int32_t) * fct.size(),
                          cudaMemcpyHostToDevice) == cudaSuccess;
    ok = ok && cudaMemcpy(h->d_fwd_class_start, fcs.data(), sizeof(int32_t) * fcs.size(),
                          cudaMemcpyHostToDevice) == cudaSuccess;
    ok = ok && cudaMemcpy(h->d_bwd_class_tables, bct.data(), sizeof(int32_t) * bct.size(),
                          cudaMemcpyHostToDevice) == cudaSuccess;
    ok = ok && cudaMemcpy(h->d_bwd_class_start, bcs.data(), sizeof(int32_t) * bcs.size(),
                          cudaMemcpyHostToDevice) == cudaSuccess;
    ok = ok && cudaMemcpy(h->d_all_tables, all.data(), sizeof(int32_t) * num_tables,
                          cudaMemcpyHostToDevice) == cudaSuccess;
    ok = ok && cudaMemcpy(h->d_all_start, all_start.data(), sizeof(int32_t) * 2,
                          cudaMemcpyHostToDevice) == cudaSuccess;
    ok = ok && cudaMemset(h->d_error, 0, sizeof(int) + sizeof(uint32_t)) == cudaSuccess;
    ok = ok && cudaMemset(h->d_zero_row, 0, 2048) == cudaSuccess;
    if (ok && (flags & CB_TIMING)) {
        for (auto& e : h->ev_fwd) ok = ok && cudaEventCreate(&e) == cudaSuccess;
        for (auto& e : h->ev_bwd) ok = ok && cudaEventCreate(&e) == cudaSuccess;
    }
    if (!ok) {
        cudaGetLastError();
        cb_tbe_destroy(h);
        return CB_ERR_CUDA;
    }
    *out = h;
    return CB_OK;
}

cb_status cb_tbe_reserve(cb_tbe* h, int32_t batch, int64_t num_indices) {
    if (!h || batch < 0 || num_indices < 0) return CB_ERR_INVALID_ARG;
    if (!current_device_ok(h)) return CB_ERR_INVALID_ARG;
    return ensure_workspace(h, batch, num_indices);
}

cb_status cb_tbe_forward(cb_tbe* h, int32_t batch, const void* indices, int64_t num_indices,
                         const void* offsets, const float* per_sample_weights, void* out,
                         cudaStream_t stream) {
    cb_status st = check_common(h, batch, indices, num_indices, offsets);
    if (st != CB_OK) return st;
    if (batch > 0 && (!out || (reinterpret_cast<uintptr_t>(out) & 15u))) return CB_ERR_INVALID_ARG;
    if (!current_device_ok(h)) return CB_ERR_INVALID_ARG;
    h->last_stream = stream;
    h->fwd_timed = false;
    if (batch == 0) return CB_OK;
    const int64_t n = num_indices;
    Problem P = make_problem(h, batch, indices, n, offsets, per_sample_weights);
    Ranges nv("cb_tbe_forward");
    nv.phase("fwd.prep");
    record(h, h->ev_fwd[0], stream);
    if (h->flags & CB_VALIDATE) {
        launch_validate_offsets(P, h->num_sms, stream);
        h->launches += 1;
    }
    if (n == 0) {
        if (cudaMemsetAsync(out, 0, static_cast<size_t>(elem_bytes(h->out_dtype)) * batch * h->sum_d, stream) !=
            cudaSuccess)
            return CB_ERR_CUDA;
        return finish_call(h, stream);
    }
    st = ensure_workspace(h, batch, n);
    if (st != CB_OK) return st;
    Workspace w;
    layout(h, batch, n, static_cast<char*>(h->ws), &w);
    Plan Q = make_plan(h, w, false, kFwdChunk);
    const int64_t bound = n / kFwdChunk + h->T + 1;
    launch_plan(P, Q, 0, nullptr, nullptr, h->num_sms, true, stream);
    h->launches += 2;
    record(h, h->ev_fwd[1], stream);
    nv.phase("fwd.gather");
    for (size_t c = 0; c < h->fwd_classes.size(); ++c) {
        launch_fwd_gather(P, Q, out, static_cast<int>(c), h->fwd_classes[c].dtype,
                          h->fwd_classes[c].vpl, h->fwd_classes[c].gc, bound, h->num_sms, stream);
        h->launches += 1;
    }
    record(h, h->ev_fwd[2], stream);
    nv.phase("fwd.fixup");
    launch_fwd_fixup(P, Q, out, bound, h->num_sms, stream);
    h->launches += 1;
    record(h, h->ev_fwd[3], stream);
    h->fwd_timed = (h->flags & CB_TIMING) != 0;
    return finish_call(h, stream);
}

cb_status cb_tbe_weight_grad(cb_tbe* h, int32_t batch, const void* indices, int64_t num_indices,
                             const void* offsets, const void* grad_out, float* grad_weights,
                             cudaStream_t stream) {
    cb_status st = check_common(h, batch, indices, num_indices, offsets);
    if (st != CB_OK) return st;
    const int64_t n = num_indices;
    if (n > 0 && batch > 0 &&
        (!grad_out || !grad_weights || (reinterpret_cast<uintptr_t>(grad_out) & 15u)))
        return CB_ERR_INVALID_ARG;
    if (!current_device_ok(h)) return CB_ERR_INVALID_ARG;
    h->last_stream = stream;
    if (n == 0 || batch == 0) return CB_OK;
    Problem P = make_problem(h, batch, indices, n, offsets, nullptr);
    if (h->flags & CB_VALIDATE) {
        launch_validate_offsets(P, h->num_sms, stream);
        h->launches += 1;
    }
    st = ensure_workspace(h, batch, n);
    if (st != CB_OK) return st;
    Workspace w;
    layout(h, batch, n, static_cast<char*>(h->ws), &w);
    Plan Q = make_plan(h, w, false, kFwdChunk);
    const int64_t bound = n / kFwdChunk + h->T + 1;
    launch_plan(P, Q, 0, nullptr, nullptr, h->num_sms, true, stream);
    h->launches += 2;
    for (size_t c = 0; c < h->fwd_classes.size(); ++c) {
        // The compiled row layouts cover one vector per lane; wider rows loop.
        const int gc = h->fwd_classes[c].vpl == 1 ? h->fwd_classes[c].gc : 0;
        launch_weight_grad(P, Q, grad_out, grad_weights, static_cast<int>(c), h->fwd_classes[c].dtype, gc,
                           bound, h->num_sms, stream);
        h->launches += 1;
    }
    return finish_call(h, stream);
}

cb_status cb_tbe_backward(cb_tbe* h, int32_t batch, const void* indices, int64_t num_indices,
                          const void* offsets, const float* per_sample_weights,
                          const void* grad_out, cb_sparse_grad* g, cudaStream_t stream) {
    if (!h) return CB_ERR_INVALID_ARG;
    if (!g || !g->table_offsets || !g->num_unique || !g->num_floats) return CB_ERR_INVALID_ARG;
    if (g->grads && (!g->unique_ids || !g->grad_offsets || g->cap_rows < 0 || g->cap_floats < 0 ||
                     (reinterpret_cast<uintptr_t>(g->grads) & 15u)))
        return CB_ERR_INVALID_ARG;
    return backward_impl(h, batch, indices, num_indices, offsets, per_sample_weights, grad_out, g, nullptr,
                         stream);
}

cb_status cb_tbe_backward_apply(cb_tbe* h, int32_t batch, const void* indices, int64_t num_indices,
                                const void* offsets, const float* per_sample_weights,
                                const void* grad_out, cb_optimizer kind, float lr, float eps,
                                float* const* state, cudaStream_t stream) {
    if (!h || !optimizer_ok(kind, lr, eps, state)) return CB_ERR_INVALID_ARG;
    ApplyArgs a;
    a.kind = kind == CB_OPT_SGD ? kApplySgd : kApplyAdagrad;
    a.lr = lr;
    a.eps = eps;
    a.state = state;
    return backward_impl(h, batch, indices, num_indices, offsets, per_sample_weights, grad_out, nullptr, &a,
                         stream);
}

cb_status cb_tbe_apply_sparse(cb_tbe* h, const cb_sparse_grad* g, cb_optimizer kind, float lr, float eps,
                              float* const* state, cudaStream_t stream) {
    if (!h || !optimizer_ok(kind, lr, eps, state)) return CB_ERR_INVALID_ARG;
    if (!g || !g->unique_ids || !g->table_offsets || !g->grad_offsets || !g->grads || !g->num_unique ||
        !g->num_floats || g->cap_rows < 0 || g->cap_floats < 0 || (reinterpret_cast<uintptr_t>(g->grads) & 15u))
        return CB_ERR_INVALID_ARG;
    if (!current_device_ok(h)) return CB_ERR_INVALID_ARG;
    h->last_stream = stream;
    const Problem P = make_problem(h, 0, nullptr, 0, nullptr, nullptr);
    BwdOut O{};
    O.unique_ids = g->unique_ids;
    O.table_offsets = g->table_offsets;
    O.grad_offsets = g->grad_offsets;
    O.grads = g->grads;
    O.cap_rows = g->cap_rows;
    O.cap_floats = g->cap_floats;
    O.num_unique = g->num_unique;
    O.num_floats = g->num_floats;
    O.apply = kind == CB_OPT_SGD ? kApplySgd : kApplyAdagrad;
    O.lr = lr;
    O.eps = eps;
    O.state = state;
    launch_apply_sparse(P, O, h->num_sms, stream);
    h->launches += 1;
    return finish_call(h, stream);
}

cb_status cb_tbe_get_error(cb_tbe* h) {
    if (!h) return CB_ERR_INVALID_ARG;
    if (cudaStreamSynchronize(h->last_stream) != cudaSuccess) {
        cudaGetLastError();
        return CB_ERR_CUDA;
    }
    int err = 0;
    if (cudaMemcpy(&err, h->d_error, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess ||
        cudaMemset(h->d_error, 0, sizeof(int)) != cudaSuccess) {
        cudaGetLastError();
        return CB_ERR_CUDA;
    }
    return static_cast<cb_status>(err);
}

cb_status cb_tbe_last_timings(cb_tbe* h, float* ms, int32_t n) {
    if (!h || !ms || n < 0 || !(h->flags & CB_TIMING)) return CB_ERR_INVALID_ARG;
    float v[kNumTimers];
    for (float& x : v) x = -1.f;
    if (h->fwd_timed) {
        if (cudaEventSynchronize(h->ev_fwd[3]) != cudaSuccess) return CB_ERR_CUDA;
        for (int i = 0; i < 3; ++i) cudaEventElapsedTime(&v[i], h->ev_fwd[i], h->ev_fwd[i + 1]);
    }
    if (h->bwd_timed) {
        if (cudaEventSynchronize(h->ev_bwd[4]) != cudaSuccess) return CB_ERR_CUDA;
        for (int i = 0; i < 4; ++i) cudaEventElapsedTime(&v[3 + i], h->ev_bwd[i], h->ev_bwd[i + 1]);
    }
    for (int i = 0; i < n && i < kNumTimers; ++i) ms[i] = v[i];
    return CB_OK;
}

uint64_t cb_tbe_launch_count(const cb_tbe* h) { return h ? h->launches : 0; }

cb_status cb_tbe_sorted_payloads(const cb_tbe* h, uint32_t* out, int64_t num_indices, cudaStream_t stream) {
    if (!h || !out || !h->last_sorted || num_indices != h->last_sorted_n) return CB_ERR_INVALID_ARG;
    if (!current_device_ok(h)) return CB_ERR_INVALID_ARG;
    if (cudaMemcpyAsync(out, h->last_sorted, sizeof(uint32_t) * num_indices, cudaMemcpyDeviceToDevice,
                        stream) != cudaSuccess) {
        cudaGetLastError();
        return CB_ERR_CUDA;
    }
    return CB_OK;
}

void cb_tbe_destroy(cb_tbe* h) {
    if (!h) return;
    cudaStreamSynchronize(h->last_stream);
    if (h->ws) cudaFree(h->ws);
    if (h->persist) cudaFree(h->persist);
    for (auto& e : h->ev_fwd)
        if (e) cudaEventDestroy(e);
    for (auto& e : h->ev_bwd)
        if (e) cudaEventDestroy(e);
    cudaGetLastError();
    delete h;
}

}  // extern "C"
