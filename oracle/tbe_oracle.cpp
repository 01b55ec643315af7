// tbe_oracle.cpp -- TEST INFRASTRUCTURE, not part of the product.
//
// A plain, slow, fp64 CPU statement of the pooled embedding-bag lookup over
// jagged categorical features and of its de-duplicated adjoint. Only tests/,
// __graft_entry__.smoke() and bench.py (cpu_baseline leg and the reference
// arm) may load this library. It shares no code, header, table or helper with
// the CUDA library under paper_2609_30656_gb300/ and never links it.
//
// What the paper fixes (Component Benchmark, arXiv 2609.30656):
//   * Abstract: the recommendation models mix memory-bandwidth-bound
//     operations with dynamic shapes that come from jagged categorical
//     features.
//   * Sec. I and Sec. III.B.1: the embedding tables are terabyte-scale and are
//     shrunk (smaller hash size) so that one GPU holds them.
//   * Sec. IV.A.2: sparse_arch performs the lookups from the embedding tables
//     and is almost entirely bandwidth-bound with low arithmetic intensity.
// The paper gives no formula for the lookup, so this file writes out the
// standard definition of a pooled embedding bag over key-major (table-major)
// jagged offsets, reading the stored table values exactly:
//
//   bag (t, b) = indices[offsets[t*B + b] .. offsets[t*B + b + 1])
//   y[b, Doff_t + j] = s_b * sum_{i in bag} w_i * E_t[indices[i], j]
//   s_b = 1 for sum pooling; 1/L for mean pooling (L = bag length; an empty
//   bag gives exact zero); w_i = per-sample weight, or 1 without weights.
//
// and its adjoint with respect to the table rows, de-duplicated per touched
// row:  G[key] = sum_{i : key_i == key} w_i * s_{b(i)} * grad_out[b(i), Doff_t ..]
// with key_i = row_base_t + indices[i]  (row_base_t = rows of tables < t).
//
// Readings where the paper is silent (each is listed in the design notes):
//   * a weighted mean divides by the bag length L, not by the sum of weights;
//   * empty bags yield exact zeros and contribute nothing to the adjoint;
//   * an index outside [0, rows_t) or malformed offsets is an error, not UB;
//   * half-precision storage widens to fp64 exactly before any arithmetic.
//
// Parity: every function here is pinned by tests/test_oracle.py against hand
// sums, closed forms, invariants and torch's CPU embedding_bag in float64.

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <new>
#include <vector>

#ifdef _OPENMP
#include <omp.h>
#endif

namespace {

// Status codes returned to the Python wrapper (independent numbering).
enum { ORC_OK = 0, ORC_BAD_ARG = 1, ORC_INDEX_OOB = 2, ORC_BAD_OFFSETS = 3 };

// Storage type codes used by the wrapper: 0 = float32, 1 = float16, 2 = bfloat16.
enum { ORC_F32 = 0, ORC_F16 = 1, ORC_BF16 = 2 };

// IEEE 754 binary16 -> double, from the format's definition: 1 sign bit,
// 5 exponent bits (bias 15), 10 fraction bits; exponent 0 encodes zero and
// subnormals (f * 2^-24), exponent 31 encodes inf / NaN.
double half_bits_to_double(uint16_t h) {
    const int sign = (h >> 15) & 1;
    const int expo = (h >> 10) & 0x1f;
    const int frac = h & 0x3ff;
    double mag;
    if (expo == 0) {
        mag = std::ldexp(static_cast<double>(frac), -24);
    } else if (expo == 31) {
        mag = frac ? NAN : INFINITY;
    } else {
        mag = std::ldexp(static_cast<double>(1024 + frac), expo - 25);
    }
    return sign ? -mag : mag;
}

// bfloat16 is the upper half of an IEEE binary32 word.
double bf16_bits_to_double(uint16_t h) {
    uint32_t w = static_cast<uint32_t>(h) << 16;
    float f;
    std::memcpy(&f, &w, sizeof f);
    return static_cast<double>(f);
}

double table_value(const void* table, int32_t dtype, int64_t flat) {
    switch (dtype) {
        case ORC_F32: return static_cast<double>(static_cast<const float*>(table)[flat]);
        case ORC_F16: return half_bits_to_double(static_cast<const uint16_t*>(table)[flat]);
        default:      return bf16_bits_to_double(static_cast<const uint16_t*>(table)[flat]);
    }
}

int64_t read_index(const void* p, int32_t is_i32, int64_t i) {
    return is_i32 ? static_cast<int64_t>(static_cast<const int32_t*>(p)[i])
                  : static_cast<const int64_t*>(p)[i];
}

// Offsets must start at 0, never decrease and end at n.
int check_offsets(const void* offsets, int32_t is_i32, int64_t num_bags, int64_t n) {
    if (read_index(offsets, is_i32, 0) != 0) return ORC_BAD_OFFSETS;
    for (int64_t k = 0; k < num_bags; ++k) {
        if (read_index(offsets, is_i32, k + 1) < read_index(offsets, is_i32, k)) return ORC_BAD_OFFSETS;
    }
    if (read_index(offsets, is_i32, num_bags) != n) return ORC_BAD_OFFSETS;
    return ORC_OK;
}

int check_indices(int32_t T, const int64_t* rows, int32_t B, const void* indices,
                  const void* offsets, int32_t is_i32) {
    for (int32_t t = 0; t < T; ++t) {
        const int64_t s = read_index(offsets, is_i32, static_cast<int64_t>(t) * B);
        const int64_t e = read_index(offsets, is_i32, static_cast<int64_t>(t + 1) * B);
        for (int64_t i = s; i < e; ++i) {
            const int64_t r = read_index(indices, is_i32, i);
            if (r < 0 || r >= rows[t]) return ORC_INDEX_OOB;
        }
    }
    return ORC_OK;
}

int check_common(int32_t T, const int64_t* rows, const int32_t* dims, int32_t B, int64_t n,
                 const void* indices, const void* offsets, int32_t is_i32) {
    if (T <= 0 || B < 0 || n < 0 || !rows || !dims || !offsets) return ORC_BAD_ARG;
    if (n > 0 && !indices) return ORC_BAD_ARG;
    for (int32_t t = 0; t < T; ++t)
        if (rows[t] < 0 || dims[t] <= 0) return ORC_BAD_ARG;
    const int64_t num_bags = static_cast<int64_t>(T) * B;
    int st = check_offsets(offsets, is_i32, num_bags, n);
    if (st != ORC_OK) return st;
    return check_indices(T, rows, B, indices, offsets, is_i32);
}

struct BackwardResult {
    int64_t num_unique = 0;
    int64_t num_floats = 0;
    std::vector<int64_t> uniq;           // ascending global ids (row_base_t + row)
    std::vector<int64_t> seg_start;      // [U + 1] start of each run in the sorted order
    std::vector<int64_t> perm;           // [n] lookup positions in sorted order
    std::vector<int64_t> table_offsets;  // [T + 1] first unique entry of each table
    std::vector<int64_t> grad_offsets;   // [U + 1] start of each row's gradient in grads
    std::vector<double> grads;           // packed rows, D_t values each
};

}  // namespace

extern "C" {

// Exposed so that the tests can pin the format decoders on every bit pattern.
double tbe_oracle_half_to_double(uint16_t h) { return half_bits_to_double(h); }
double tbe_oracle_bf16_to_double(uint16_t h) { return bf16_bits_to_double(h); }

// Forward: out[b, Doff_t + j] for every table t and bag b (row-major [B, sum D]).
// threads <= 0 uses the OpenMP default; bags are independent, so the loop over
// them may run in parallel without changing any result.
int tbe_oracle_forward(int32_t T, const int64_t* rows, const int32_t* dims, const int32_t* dtypes,
                       const void* const* tables, int32_t B, const void* indices, int32_t idx_is_i32,
                       int64_t n, const void* offsets, const float* weights, int32_t mean_pooling,
                       int32_t threads, double* out) {
    int st = check_common(T, rows, dims, B, n, indices, offsets, idx_is_i32);
    if (st != ORC_OK) return st;
    if (!out || !dtypes || !tables) return ORC_BAD_ARG;

    std::vector<int64_t> doff(T + 1, 0);
    for (int32_t t = 0; t < T; ++t) doff[t + 1] = doff[t] + dims[t];
    const int64_t sum_d = doff[T];
    const int64_t num_bags = static_cast<int64_t>(T) * B;

#ifdef _OPENMP
    const int nthr = threads > 0 ? threads : omp_get_max_threads();
#pragma omp parallel for schedule(dynamic, 16) num_threads(nthr)
#endif
    for (int64_t bag = 0; bag < num_bags; ++bag) {
        const int32_t t = static_cast<int32_t>(bag / B);
        const int64_t b = bag % B;
        const int32_t D = dims[t];
        const int64_t s = read_index(offsets, idx_is_i32, bag);
        const int64_t e = read_index(offsets, idx_is_i32, bag + 1);
        const int64_t L = e - s;
        std::vector<double> acc(D, 0.0);
        for (int64_t i = s; i < e; ++i) {
            const int64_t r = read_index(indices, idx_is_i32, i);
            const double w = weights ? static_cast<double>(weights[i]) : 1.0;
            for (int32_t j = 0; j < D; ++j)
                acc[j] += w * table_value(tables[t], dtypes[t], r * D + j);
        }
        if (mean_pooling && L > 0)
            for (int32_t j = 0; j < D; ++j) acc[j] /= static_cast<double>(L);
        double* y = out + b * sum_d + doff[t];
        for (int32_t j = 0; j < D; ++j) y[j] = acc[j];
    }
    return ORC_OK;
}

// Gradient with respect to the per-sample weights. The output is linear in
// each w_i, so d<grad_out, y>/d w_i = s_b * sum_j grad_out[b, Doff_t + j] *
// E_t[indices[i], j] (s_b = 1/L for mean pooling, 1 for sum), whatever the
// weights are; out is [n] in lookup order.
int tbe_oracle_weight_grad(int32_t T, const int64_t* rows, const int32_t* dims, const int32_t* dtypes,
                           const void* const* tables, int32_t B, const void* indices,
                           int32_t idx_is_i32, int64_t n, const void* offsets, int32_t mean_pooling,
                           const float* grad_out, int32_t threads, double* out) {
    int st = check_common(T, rows, dims, B, n, indices, offsets, idx_is_i32);
    if (st != ORC_OK) return st;
    if ((n > 0 && !out) || !dtypes || !tables || (n > 0 && B > 0 && !grad_out)) return ORC_BAD_ARG;

    std::vector<int64_t> doff(T + 1, 0);
    for (int32_t t = 0; t < T; ++t) doff[t + 1] = doff[t] + dims[t];
    const int64_t sum_d = doff[T];
    const int64_t num_bags = static_cast<int64_t>(T) * B;

#ifdef _OPENMP
    const int nthr = threads > 0 ? threads : omp_get_max_threads();
#pragma omp parallel for schedule(dynamic, 16) num_threads(nthr)
#endif
    for (int64_t bag = 0; bag < num_bags; ++bag) {
        const int32_t t = static_cast<int32_t>(bag / B);
        const int64_t b = bag % B;
        const int32_t D = dims[t];
        const int64_t s = read_index(offsets, idx_is_i32, bag);
        const int64_t e = read_index(offsets, idx_is_i32, bag + 1);
        const double scale = mean_pooling && e > s ? 1.0 / static_cast<double>(e - s) : 1.0;
        const float* g = grad_out + b * sum_d + doff[t];
        for (int64_t i = s; i < e; ++i) {
            const int64_t r = read_index(indices, idx_is_i32, i);
            double dot = 0.0;
            for (int32_t j = 0; j < D; ++j)
                dot += static_cast<double>(g[j]) * table_value(tables[t], dtypes[t], r * D + j);
            out[i] = scale * dot;
        }
    }
    return ORC_OK;
}

// Backward, de-duplicated: stable comparison sort of (key, position) by key,
// runs of equal keys, then one fp64 sum per run in ascending position order.
// The result is held in an opaque object; fetch it with the calls below.
void* tbe_oracle_backward_run(int32_t T, const int64_t* rows, const int32_t* dims, int32_t B,
                              const void* indices, int32_t idx_is_i32, int64_t n, const void* offsets,
                              const float* weights, int32_t mean_pooling, const float* grad_out,
                              int32_t threads, int32_t* status) {
    int st = check_common(T, rows, dims, B, n, indices, offsets, idx_is_i32);
    if (st == ORC_OK && n > 0 && !grad_out) st = ORC_BAD_ARG;
    if (status) *status = st;
    if (st != ORC_OK) return nullptr;

    auto* res = new (std::nothrow) BackwardResult();
    if (!res) {
        if (status) *status = ORC_BAD_ARG;
        return nullptr;
    }
    std::vector<int64_t> doff(T + 1, 0), row_base(T + 1, 0);
    for (int32_t t = 0; t < T; ++t) {
        doff[t + 1] = doff[t] + dims[t];
        row_base[t + 1] = row_base[t] + rows[t];
    }
    const int64_t sum_d = doff[T];

    // Step 1: the lookup list with its table, bag, key and coefficient w_i * s_b.
    std::vector<int64_t> key(n), bag_of(n);
    std::vector<int32_t> table_of(n);
    std::vector<double> coef(n);
    for (int32_t t = 0; t < T; ++t) {
        for (int64_t b = 0; b < B; ++b) {
            const int64_t bag = static_cast<int64_t>(t) * B + b;
            const int64_t s = read_index(offsets, idx_is_i32, bag);
            const int64_t e = read_index(offsets, idx_is_i32, bag + 1);
            for (int64_t i = s; i < e; ++i) {
                key[i] = row_base[t] + read_index(indices, idx_is_i32, i);
                bag_of[i] = b;
                table_of[i] = t;
                const double w = weights ? static_cast<double>(weights[i]) : 1.0;
                coef[i] = mean_pooling ? w / static_cast<double>(e - s) : w;
            }
        }
    }

    // Step 2: stable sort of positions by key (ties keep ascending position).
    res->perm.resize(n);
    for (int64_t i = 0; i < n; ++i) res->perm[i] = i;
    std::stable_sort(res->perm.begin(), res->perm.end(),
                     [&](int64_t a, int64_t b) { return key[a] < key[b]; });

    // Step 3: runs of equal keys.
    for (int64_t k = 0; k < n; ++k) {
        if (k == 0 || key[res->perm[k]] != key[res->perm[k - 1]]) {
            res->uniq.push_back(key[res->perm[k]]);
            res->seg_start.push_back(k);
        }
    }
    res->num_unique = static_cast<int64_t>(res->uniq.size());
    res->seg_start.push_back(n);

    // Per-table ranges of unique entries and packed gradient offsets.
    res->table_offsets.assign(T + 1, 0);
    for (int32_t t = 0; t <= T; ++t)
        res->table_offsets[t] = std::lower_bound(res->uniq.begin(), res->uniq.end(), row_base[t]) -
                                res->uniq.begin();
    res->grad_offsets.assign(res->num_unique + 1, 0);
    for (int64_t u = 0; u < res->num_unique; ++u) {
        const int32_t t = static_cast<int32_t>(
            std::upper_bound(row_base.begin(), row_base.end(), res->uniq[u]) - row_base.begin() - 1);
        res->grad_offsets[u + 1] = res->grad_offsets[u] + dims[t];
    }
    res->num_floats = res->grad_offsets[res->num_unique];
    res->grads.assign(static_cast<size_t>(res->num_floats), 0.0);

    // Step 4: one fp64 sum per run, in ascending position order.
#ifdef _OPENMP
    const int nthr = threads > 0 ? threads : omp_get_max_threads();
#pragma omp parallel for schedule(dynamic, 64) num_threads(nthr)
#endif
    for (int64_t u = 0; u < res->num_unique; ++u) {
        double* g = res->grads.data() + res->grad_offsets[u];
        for (int64_t k = res->seg_start[u]; k < res->seg_start[u + 1]; ++k) {
            const int64_t i = res->perm[k];
            const int32_t t = table_of[i];
            const float* go = grad_out + bag_of[i] * sum_d + doff[t];
            for (int32_t j = 0; j < dims[t]; ++j) g[j] += coef[i] * static_cast<double>(go[j]);
        }
    }
    return res;
}

int64_t tbe_oracle_backward_num_unique(const void* r) {
    return static_cast<const BackwardResult*>(r)->num_unique;
}
int64_t tbe_oracle_backward_num_floats(const void* r) {
    return static_cast<const BackwardResult*>(r)->num_floats;
}

// Copies the result out. Each destination may be null; sizes are
// uniq [U], seg_start [U + 1], perm [n], table_offsets [T + 1],
// grad_offsets [U + 1], grads [num_floats].
void tbe_oracle_backward_fetch(const void* r, int64_t* uniq, int64_t* seg_start, int64_t* perm,
                               int64_t* table_offsets, int64_t* grad_offsets, double* grads) {
    const auto* res = static_cast<const BackwardResult*>(r);
    auto copy = [](const auto& v, auto* dst) {
        if (dst && !v.empty()) std::memcpy(dst, v.data(), v.size() * sizeof(v[0]));
    };
    copy(res->uniq, uniq);
    copy(res->seg_start, seg_start);
    copy(res->perm, perm);
    copy(res->table_offsets, table_offsets);
    copy(res->grad_offsets, grad_offsets);
    copy(res->grads, grads);
}

void tbe_oracle_backward_free(void* r) { delete static_cast<BackwardResult*>(r); }

// Dense adjoint by direct scatter-add, the plain transpose of the forward map:
//   dE_t[indices[i], :] += w_i * s_b * grad_out[b, Doff_t : Doff_t + D_t]
// for every lookup i of bag (t, b). It does not sort, so it is an independent
// statement of the same quantity as the de-duplicated backward.
// dense[t] points to a [rows_t, D_t] fp64 buffer that this call zero-fills.
int tbe_oracle_backward_dense(int32_t T, const int64_t* rows, const int32_t* dims, int32_t B,
                              const void* indices, int32_t idx_is_i32, int64_t n, const void* offsets,
                              const float* weights, int32_t mean_pooling, const float* grad_out,
                              double* const* dense) {
    int st = check_common(T, rows, dims, B, n, indices, offsets, idx_is_i32);
    if (st != ORC_OK) return st;
    if (!dense || (n > 0 && !grad_out)) return ORC_BAD_ARG;
    int64_t sum_d = 0;
    for (int32_t t = 0; t < T; ++t) sum_d += dims[t];
    int64_t doff = 0;
    for (int32_t t = 0; t < T; ++t) {
        const int32_t D = dims[t];
        std::fill(dense[t], dense[t] + rows[t] * D, 0.0);
        for (int64_t b = 0; b < B; ++b) {
            const int64_t bag = static_cast<int64_t>(t) * B + b;
            const int64_t s = read_index(offsets, idx_is_i32, bag);
            const int64_t e = read_index(offsets, idx_is_i32, bag + 1);
            for (int64_t i = s; i < e; ++i) {
                const int64_t r = read_index(indices, idx_is_i32, i);
                double c = weights ? static_cast<double>(weights[i]) : 1.0;
                if (mean_pooling) c /= static_cast<double>(e - s);
                const float* go = grad_out + b * sum_d + doff;
                for (int32_t j = 0; j < D; ++j) dense[t][r * D + j] += c * static_cast<double>(go[j]);
            }
        }
        doff += D;
    }
    return ORC_OK;
}

}  // extern "C"
