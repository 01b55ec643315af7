// fm_oracle.cpp -- TEST INFRASTRUCTURE, not part of the product.
//
// A plain fp64 CPU statement of the factorization-machine cross term on the
// pooled embeddings, the step that follows the lookups in the paper's
// DeepFM-based model (Sec. IV.A.2: inter_arch.fm computes the factorization
// machine's cross term, bandwidth-bound, a few element-wise and reduction
// passes). The paper gives no formula; this file writes out the pairwise
// definition of the second-order term of the factorization machine (Rendle,
// 2010, which the paper cites), with each table's pooled row as one field
// embedding:
//
//   v_{b,t} = y[b, t*D : (t+1)*D]                    (T fields, D columns)
//   fm[b]   = sum_{t < u} <v_{b,t}, v_{b,u}>
//
// and its gradient with respect to the pooled rows, times an upstream
// gradient g[b]:
//
//   d fm[b] / d y[b, t*D + j] = sum_{u != t} y[b, u*D + j]
//   grad_y[b, t*D + j] = g[b] * sum_{u != t} y[b, u*D + j]
//
// Both are the definitions themselves, O(T^2 D) per sample, with no
// rewriting; tests/test_oracle.py pins them to the closed form
// 1/2 [(sum v)^2 - sum v^2], to exact finite differences of this quadratic,
// and to small cases worked by hand. Only tests/ and bench.py may load it.

#include <cstdint>

extern "C" {

// y: [B, row_stride] fp32, fields t at columns [t*D, (t+1)*D). out: [B] fp64.
int fm_oracle_forward(int32_t B, int32_t T, int32_t D, int64_t row_stride, const float* y,
                      double* out) {
    if (B < 0 || T < 0 || D < 0 || row_stride < static_cast<int64_t>(T) * D) return 1;
    if (B > 0 && (!y || !out)) return 1;
#pragma omp parallel for schedule(static)
    for (int64_t b = 0; b < B; ++b) {
        const float* row = y + b * row_stride;
        double acc = 0.0;
        for (int32_t t = 0; t < T; ++t)
            for (int32_t u = t + 1; u < T; ++u) {
                double dot = 0.0;
                for (int32_t j = 0; j < D; ++j)
                    dot += static_cast<double>(row[t * D + j]) * static_cast<double>(row[u * D + j]);
                acc += dot;
            }
        out[b] = acc;
    }
    return 0;
}

// g: [B] fp32 upstream gradient. grad_y: [B, T*D] fp64 (dense, no stride).
int fm_oracle_backward(int32_t B, int32_t T, int32_t D, int64_t row_stride, const float* y,
                       const float* g, double* grad_y) {
    if (B < 0 || T < 0 || D < 0 || row_stride < static_cast<int64_t>(T) * D) return 1;
    if (B > 0 && (!y || !g || !grad_y)) return 1;
#pragma omp parallel for schedule(static)
    for (int64_t b = 0; b < B; ++b) {
        const float* row = y + b * row_stride;
        double* out = grad_y + b * static_cast<int64_t>(T) * D;
        for (int32_t t = 0; t < T; ++t)
            for (int32_t j = 0; j < D; ++j) {
                double others = 0.0;
                for (int32_t u = 0; u < T; ++u)
                    if (u != t) others += static_cast<double>(row[u * D + j]);
                out[t * D + j] = static_cast<double>(g[b]) * others;
            }
    }
    return 0;
}

}  // extern "C"
