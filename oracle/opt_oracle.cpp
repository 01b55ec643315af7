// opt_oracle.cpp -- TEST INFRASTRUCTURE, not part of the product.
//
// A plain fp64 CPU statement of a row-wise optimizer step applied to the rows
// that the de-duplicated backward touched. The paper frames its benchmark as a
// training-time tool (Sec. I, Sec. III); it names no optimizer, so this file
// writes out the two standard sparse updates of embedding training, one per
// touched row r of table t with gradient row G (the oracle's de-duplicated
// adjoint, fp64):
//
//   SGD:                E[r, j] <- round_S(E[r, j] - lr * G[j])
//   row-wise Adagrad:   m[r]    <- round_f32(m[r] + (1/D) * sum_j G[j]^2)
//                       E[r, j] <- round_S(E[r, j] - lr * G[j] / (sqrt(m[r]) + eps))
//
// with the new m[r] taken in fp64 before it is rounded for storage, and
// round_S the round-to-nearest-even conversion of the fp64 result to the
// table's storage type. The conversions are written from the formats'
// definitions below; tests/test_opt_oracle.py pins them on every bit pattern.
// Only tests/ and bench.py may load this library.

#include <cmath>
#include <cstdint>
#include <cstring>

namespace {

enum { OPT_F32 = 0, OPT_F16 = 1, OPT_BF16 = 2 };

// A finite double magnitude a >= 0 rounded to nearest-even on a binary format
// with `mant` fraction bits, minimum normal exponent emin and maximum exponent
// emax. Returns the encoded bits (exponent field << mant | fraction), or the
// infinity encoding when the rounded value overflows.
uint32_t round_to_format(double a, int mant, int emin, int emax) {
    const int bias = -emin + 1;
    const uint32_t inf = static_cast<uint32_t>(emax + bias + 1) << mant;
    if (a == 0.0) return 0;
    int e2;
    std::frexp(a, &e2);      // a = f * 2^e2, f in [0.5, 1)
    int E = e2 - 1;          // a in [2^E, 2^(E+1))
    if (E < emin) {          // subnormal range: quantum 2^(emin - mant)
        const double q = std::nearbyint(std::ldexp(a, mant - emin));  // exact scaling, then RNE
        return static_cast<uint32_t>(q);  // q == 2^mant is the smallest normal, as encoded
    }
    double q = std::nearbyint(std::ldexp(a, mant - E));  // in [2^mant, 2^(mant+1)]
    if (q == std::ldexp(1.0, mant + 1)) {
        q = std::ldexp(1.0, mant);
        ++E;
    }
    if (E > emax) return inf;
    return (static_cast<uint32_t>(E + bias) << mant) | (static_cast<uint32_t>(q) - (1u << mant));
}

uint16_t double_to_half(double x) {
    const uint16_t sign = std::signbit(x) ? 0x8000 : 0;
    if (std::isnan(x)) return 0x7e00;
    if (std::isinf(x)) return sign | 0x7c00;
    return sign | static_cast<uint16_t>(round_to_format(std::fabs(x), 10, -14, 15));
}

uint16_t double_to_bf16(double x) {
    const uint16_t sign = std::signbit(x) ? 0x8000 : 0;
    if (std::isnan(x)) return 0x7fc0;
    if (std::isinf(x)) return sign | 0x7f80;
    return sign | static_cast<uint16_t>(round_to_format(std::fabs(x), 7, -126, 127));
}

double half_to_double(uint16_t h) {
    const int e = (h >> 10) & 0x1f, f = h & 0x3ff;
    double m = e == 0 ? std::ldexp(static_cast<double>(f), -24)
             : e == 31 ? (f ? NAN : INFINITY)
                       : std::ldexp(static_cast<double>(1024 + f), e - 25);
    return (h & 0x8000) ? -m : m;
}

double bf16_to_double(uint16_t h) {
    const uint32_t w = static_cast<uint32_t>(h) << 16;
    float f;
    std::memcpy(&f, &w, sizeof f);
    return f;
}

double load(const void* p, int dtype, int64_t k) {
    if (dtype == OPT_F32) return static_cast<const float*>(p)[k];
    const uint16_t h = static_cast<const uint16_t*>(p)[k];
    return dtype == OPT_F16 ? half_to_double(h) : bf16_to_double(h);
}

void store(void* p, int dtype, int64_t k, double v) {
    if (dtype == OPT_F32) static_cast<float*>(p)[k] = static_cast<float>(v);  // RNE
    else if (dtype == OPT_F16) static_cast<uint16_t*>(p)[k] = double_to_half(v);
    else static_cast<uint16_t*>(p)[k] = double_to_bf16(v);
}

}  // namespace

extern "C" {

uint16_t opt_oracle_double_to_half(double x) { return double_to_half(x); }
uint16_t opt_oracle_double_to_bf16(double x) { return double_to_bf16(x); }

// Applies the step to every touched row. uniq [U] are global row ids
// (row_base_t + r), ascending; grad_offsets [U + 1] index the fp64 gradient
// rows in grads. tables / dtypes / dims / rows describe the T tables (updated
// in place); state [T] points at fp32 [rows_t] (row-wise Adagrad only).
// kind: 0 = SGD, 1 = row-wise Adagrad. Returns 0, or 1 on a bad argument.
int opt_oracle_apply(int32_t T, void* const* tables, const int32_t* dtypes, const int32_t* dims,
                     const int64_t* rows, int64_t U, const int64_t* uniq, const int64_t* grad_offsets,
                     const double* grads, int32_t kind, double lr, double eps, float* const* state) {
    if (T < 1 || U < 0 || (kind != 0 && kind != 1) || (kind == 1 && !state)) return 1;
    int64_t base = 0;
    int32_t t = 0;
    for (int64_t u = 0; u < U; ++u) {
        while (t < T && uniq[u] >= base + rows[t]) base += rows[t++];
        if (t >= T) return 1;
        const int64_t r = uniq[u] - base;
        const int32_t D = dims[t];
        const double* G = grads + grad_offsets[u];
        double scale = lr;
        if (kind == 1) {
            double sq = 0.0;
            for (int32_t j = 0; j < D; ++j) sq += G[j] * G[j];
            const double m = static_cast<double>(state[t][r]) + sq / D;
            state[t][r] = static_cast<float>(m);
            scale = lr / (std::sqrt(m) + eps);
        }
        for (int32_t j = 0; j < D; ++j) {
            const int64_t k = r * D + j;
            store(tables[t], dtypes[t], k, load(tables[t], dtypes[t], k) - scale * G[j]);
        }
    }
    return 0;
}

}  // extern "C"
