// cb_tbe_noalloc.cu -- cb_tbe_forward_noalloc: the forward lookup for callers
// that must not allocate device memory.
//
// Some host programs cannot call cudaMalloc once they are running: a plugin
// inside an inference server whose framework owns every byte of device memory,
// or a latency-critical loop in which an allocation (and the device-wide
// synchronisation a cudaFree brings) is not allowed. This entry point needs
// neither a handle nor a workspace: its scratch (table descriptors, the chunk
// plan and the partial sums of bags split across chunks) lives in one
// file-scope __device__ array of fixed size, which every GPU that loads this
// library holds until the process exits. The kernels are the same ones the
// handle-based forward launches.
#include <cstdint>
#include <cstring>
#include <mutex>
#include <vector>

#include "cb_tbe.h"
#include "tbe_internal.cuh"
#include "tbe_launch.h"

using namespace cbtbe;

namespace {

constexpr size_t kScratchBytes = size_t(16) << 20;  // 16 MiB per device
constexpr int64_t kChunk = 512;                      // lookups per chunk, as in the handle path
constexpr int kMaxDevices = 64;

__device__ __align__(256) unsigned char g_scratch[kScratchBytes];

std::mutex g_mutex;
void* g_scratch_addr[kMaxDevices] = {};

// The array's name is only a host-side stand-in; kernels need its device
// address, looked up once per device with that device current.
cb_status scratch_address(int device, unsigned char** out) {
    if (device < 0 || device >= kMaxDevices) return CB_ERR_INVALID_ARG;
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!g_scratch_addr[device]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || !p) {
            cudaGetLastError();
            return CB_ERR_CUDA;
        }
        g_scratch_addr[device] = p;
    }
    *out = static_cast<unsigned char*>(g_scratch_addr[device]);
    return CB_OK;
}

size_t up256(size_t x) { return (x + 255) & ~size_t(255); }

void split(int vecs, int32_t* lanes, int32_t* groups) {
    if (vecs >= 32) {
        *lanes = 32;
        *groups = 1;
    } else if ((vecs & (vecs - 1)) == 0) {
        *lanes = vecs;
        *groups = 32 / vecs;
    } else {
        *lanes = vecs;
        *groups = 1;
    }
}

}  // namespace

extern "C" cb_status cb_tbe_forward_noalloc(const cb_table_desc* tables, int32_t num_tables,
                                            cb_pooling mode, cb_index_dtype idx_dtype,
                                            int32_t batch, const void* indices,
                                            int64_t num_indices, const void* offsets,
                                            const float* per_sample_weights, float* out,
                                            cudaStream_t stream) {
    if (!tables || num_tables <= 0 || batch < 0 || num_indices < 0 || !offsets ||
        (num_indices > 0 && !indices))
        return CB_ERR_INVALID_ARG;
    if (mode != CB_POOL_SUM && mode != CB_POOL_MEAN) return CB_ERR_INVALID_ARG;
    if (idx_dtype != CB_I32 && idx_dtype != CB_I64) return CB_ERR_INVALID_ARG;
    if (static_cast<int64_t>(num_tables) * batch >= (int64_t(1) << 31)) return CB_ERR_INVALID_ARG;
    if (batch > 0 && (!out || (reinterpret_cast<uintptr_t>(out) & 15u))) return CB_ERR_INVALID_ARG;

    // Table descriptors and kernel classes, exactly as cb_tbe_create builds them.
    std::vector<TableDev> td(num_tables);
    struct Cls { int dtype, vpl, gc; std::vector<int32_t> t; };
    std::vector<Cls> classes;
    int64_t row_base = 0, doff = 0;
    int32_t dmax = 0;
    for (int32_t t = 0; t < num_tables; ++t) {
        const cb_table_desc& d = tables[t];
        const bool dt_ok = d.dtype == CB_F32 || d.dtype == CB_F16 || d.dtype == CB_BF16;
        if (!dt_ok || d.rows < 0 || d.dim <= 0 || d.dim > 512 || (d.rows > 0 && !d.data) ||
            (reinterpret_cast<uintptr_t>(d.data) & 15u))
            return CB_ERR_INVALID_ARG;
        const int64_t row_bytes = static_cast<int64_t>(d.dim) * (d.dtype == CB_F32 ? 4 : 2);
        if (row_bytes % 16 != 0) return CB_ERR_INVALID_ARG;
        TableDev& x = td[t];
        x = TableDev{};
        x.data = d.data;
        x.rows = d.rows;
        x.row_base = row_base;
        x.key_base = row_base + t;
        x.dim = d.dim;
        x.doff = static_cast<int32_t>(doff);
        x.dtype = d.dtype;
        x.row_vecs = static_cast<int32_t>(row_bytes / 16);
        split(x.row_vecs, &x.lanes, &x.groups);
        x.grad_vecs = d.dim / 4;
        split(x.grad_vecs, &x.grad_lanes, &x.grad_groups);
        const int vpl = x.row_vecs <= 32 ? 1 : (x.row_vecs <= 64 ? 2 : 4);
        const int gc = compile_time_groups(vpl, x.lanes, x.groups);
        int c = -1;
        for (size_t k = 0; k < classes.size(); ++k)
            if (classes[k].dtype == d.dtype && classes[k].vpl == vpl && classes[k].gc == gc)
                c = static_cast<int>(k);
        if (c < 0) {
            classes.push_back({d.dtype, vpl, gc, {}});
            c = static_cast<int>(classes.size() - 1);
        }
        classes[c].t.push_back(t);
        x.fwd_class = c;
        row_base += d.rows;
        doff += d.dim;
        dmax = d.dim > dmax ? d.dim : dmax;
    }
    if (row_base >= (int64_t(1) << 32) || doff >= (int64_t(1) << 31)) return CB_ERR_INVALID_ARG;
    std::vector<int32_t> class_tables, class_start{0};
    for (auto& c : classes) {
        class_tables.insert(class_tables.end(), c.t.begin(), c.t.end());
        class_start.push_back(static_cast<int32_t>(class_tables.size()));
    }

    // Layout of the static scratch for this call; refuse calls that do not fit.
    const int64_t T = num_tables, nc = static_cast<int64_t>(classes.size());
    const int64_t max_chunks = num_indices / kChunk + T + 1;
    // Each chunk takes a descriptor, an owner word and two carry rows; refuse a
    // call whose chunks alone exceed the array before any product below can
    // wrap around (num_indices near 2^63).
    const size_t per_chunk = sizeof(Chunk) + sizeof(int64_t) + 2 * sizeof(float) * static_cast<size_t>(dmax);
    if (max_chunks > static_cast<int64_t>(kScratchBytes / per_chunk)) return CB_ERR_CAPACITY;
    size_t off = 0;
    const size_t o_err = off; off += up256(sizeof(int));
    const size_t o_zero = off; off += up256(2048);
    const size_t o_tab = off; off += up256(sizeof(TableDev) * T);
    const size_t o_ct = off; off += up256(sizeof(int32_t) * T);
    const size_t o_cs = off; off += up256(sizeof(int32_t) * (nc + 1));
    const size_t o_pos = off; off += up256(sizeof(int64_t) * (T + 1));
    const size_t o_ord = off; off += up256(sizeof(int64_t) * (T + 1));
    const size_t o_cb = off; off += up256(sizeof(int64_t) * (nc + 1));
    const size_t o_ch = off; off += up256(sizeof(Chunk) * max_chunks);
    const size_t o_hd = off; off += up256(sizeof(float) * max_chunks * dmax);
    const size_t o_tl = off; off += up256(sizeof(float) * max_chunks * dmax);
    const size_t o_to = off; off += up256(sizeof(int64_t) * max_chunks);
    const size_t o_nx = off; off += up256(sizeof(uint32_t) * (nc + 1));  // chunk counters
    if (off > kScratchBytes) return CB_ERR_CAPACITY;

    int device = -1;
    if (cudaGetDevice(&device) != cudaSuccess) {
        cudaGetLastError();
        return CB_ERR_CUDA;
    }
    unsigned char* base = nullptr;
    cb_status st = scratch_address(device, &base);
    if (st != CB_OK) return st;
    if (batch == 0) return CB_OK;

    // The array keeps the previous call's contents: upload this call's tables
    // and class lists, and clear the error word and the zero row, which must
    // start at zero.
    std::vector<unsigned char> host(o_pos - o_tab, 0);
    memcpy(host.data(), td.data(), sizeof(TableDev) * T);
    memcpy(host.data() + (o_ct - o_tab), class_tables.data(), sizeof(int32_t) * T);
    memcpy(host.data() + (o_cs - o_tab), class_start.data(), sizeof(int32_t) * (nc + 1));
    if (cudaMemcpyAsync(base + o_tab, host.data(), host.size(), cudaMemcpyHostToDevice, stream) !=
            cudaSuccess ||
        cudaMemsetAsync(base + o_err, 0, sizeof(int), stream) != cudaSuccess ||
        cudaMemsetAsync(base + o_zero, 0, 2048, stream) != cudaSuccess) {
        cudaGetLastError();
        return CB_ERR_CUDA;
    }

    Problem P;
    P.tables = reinterpret_cast<const TableDev*>(base + o_tab);
    P.zero_row = reinterpret_cast<const uint4*>(base + o_zero);
    P.indices = indices;
    P.offsets = offsets;
    P.weights = per_sample_weights;
    P.error = reinterpret_cast<int*>(base + o_err);
    P.n = num_indices;
    P.T = num_tables;
    P.B = batch;
    P.sum_d = static_cast<int32_t>(doff);
    P.is32 = idx_dtype == CB_I32;
    P.mean = mode == CB_POOL_MEAN;
    P.dmax = dmax;
    P.out_dtype = CB_F32;
    int num_sms = 1;
    cudaDeviceGetAttribute(&num_sms, cudaDevAttrMultiProcessorCount, device);
    launch_validate_offsets(P, num_sms, stream);
    if (num_indices == 0) {
        if (cudaMemsetAsync(out, 0, sizeof(float) * batch * doff, stream) != cudaSuccess) {
            cudaGetLastError();
            return CB_ERR_CUDA;
        }
    } else {
        Plan Q;
        Q.chunk_len = static_cast<int32_t>(kChunk);
        Q.snap_cap = static_cast<int32_t>(4 * kChunk);  // as the handle's forward
        Q.num_classes = static_cast<int32_t>(nc);
        Q.class_tables = reinterpret_cast<const int32_t*>(base + o_ct);
        Q.class_table_start = reinterpret_cast<const int32_t*>(base + o_cs);
        Q.table_pos = reinterpret_cast<int64_t*>(base + o_pos);
        Q.ord_chunk_base = reinterpret_cast<int64_t*>(base + o_ord);
        Q.class_chunk_base = reinterpret_cast<int64_t*>(base + o_cb);
        Q.chunks = reinterpret_cast<Chunk*>(base + o_ch);
        Q.max_chunks = max_chunks;
        Q.carry_head = reinterpret_cast<float*>(base + o_hd);
        Q.carry_tail = reinterpret_cast<float*>(base + o_tl);
        Q.tail_owner = reinterpret_cast<int64_t*>(base + o_to);
        Q.chunk_next = reinterpret_cast<uint32_t*>(base + o_nx);  // zeroed by the plan
        launch_plan(P, Q, 0, nullptr, nullptr, num_sms, true, stream);
        for (size_t c = 0; c < classes.size(); ++c)
            launch_fwd_gather(P, Q, out, static_cast<int>(c), classes[c].dtype, classes[c].vpl,
                              classes[c].gc, max_chunks, num_sms, stream);
        launch_fwd_fixup(P, Q, out, max_chunks, num_sms, stream);
    }
    if (cudaGetLastError() != cudaSuccess) return CB_ERR_CUDA;
    int err = 0;
    if (cudaMemcpyAsync(&err, base + o_err, sizeof(int), cudaMemcpyDeviceToHost, stream) !=
            cudaSuccess ||
        cudaStreamSynchronize(stream) != cudaSuccess) {
        cudaGetLastError();
        return CB_ERR_CUDA;
    }
    return static_cast<cb_status>(err);
}
