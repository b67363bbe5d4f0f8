// pps_device.cuh -- device primitives of the keyed Poisson race (sm_103a).
//
// Keyed source: Philox4x32-10 (Salmon et al., SC'11) evaluated in registers,
// one block of four 32-bit words per four consecutive tokens.  Counter
// (token >> 2, pos, ctx_lo, ctx_hi), key (key_lo ^ (j-1) * 0x9E3779B9, key_hi)
// for arrival j; the word of token i is lane i & 3.  u = (w + 1/2) 2^-32,
// E = -ln u (first arrival scaled to Exp(1), Thm A.1).
//
// Keys.  The streaming kernels order tokens by the fp32 key
//     k(i) = log2(-log2 u_i) - logit_i * log2(e) / T
//          = log2(e) * (ln E_i - logit_i / T) + log2(log2 e),
// an increasing affine map of the paper's race key s = ln E - l/T (Alg. 2,
// App. A.2), so the order and the argmin are the same.  The fp32 value carries
// an error bounded by key_err_bound(); pairs closer than the sum of their
// bounds are re-ordered with the fp64 key s.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>
#include "pps_internal.h"

namespace pps {

constexpr uint32_t kPhiloxM0 = 0xD2511F53u;
constexpr uint32_t kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u;
constexpr uint32_t kPhiloxW1 = 0xBB67AE85u;

constexpr float kLog2e = 1.4426950408889634f;
constexpr double kLn2 = 0.69314718055994530942;
// log2(ln 2): converts the filter bound E < 2^(theta + l c) ln 2 into base-2 exponents
constexpr float kLog2Ln2 = -0.52876637294589f;
// bound on |k_fp32 - k_exact| is kErrAbs + kErrRel * (|k| + kErrSpan); the
// self-test measures the transform part (largest |x32 - x64| over all 2^32 words)
constexpr float kErrAbs = 3.0e-6f;
constexpr float kErrRel = 1.2e-7f;  // ~2^-23: rounding of c = log2(e)/T and of the fused multiply-add
constexpr float kErrSpan = 40.0f;   // |log2(-log2 u)| <= 34.9 for every 32-bit word
// the filter may only drop a token whose fp32 key is >= theta; it tests
// E >= v with theta raised by this margin (log2 units), which covers the
// approximate ex2, the rounding of z and the key error for |theta| < 2^16
constexpr float kFilterMargin = 0.015625f;

__device__ __forceinline__ float key_err_bound(float k) { return kErrAbs + kErrRel * (fabsf(k) + kErrSpan); }

// Filter bound for a list whose k-th key is t: t plus four error bounds, so
// that a row's k-th key tau <= t and a drop bound of filter_slack(t) always
// pass the completeness test tau + err(tau) + err(bound) < bound (|tau| grows
// by at most t - tau, and err by kErrRel times that).  +inf stays +inf.
__device__ __forceinline__ float filter_slack(float t) { return t + 4.0f * key_err_bound(t); }

// ------------------------------------------------------------------ Philox
//
// PPS_PHILOX_ROUNDS: rounds of the keyed source's Philox4x32.  10 (Salmon et
// al.'s default) unless the library is built with 7, the smallest count they
// report free of Crush failures (libpps_r7.so; pps_philox_rounds() tells a
// caller which one it loaded).
static_assert(PPS_PHILOX_ROUNDS >= 3 && PPS_PHILOX_ROUNDS <= 16, "two hoisted rounds and at least one more");

__device__ __forceinline__ void mulhilo(uint32_t a, uint32_t b, uint32_t& hi, uint32_t& lo) {
    uint64_t p = (uint64_t)a * (uint64_t)b;
    hi = (uint32_t)(p >> 32);
    lo = (uint32_t)p;
}

// full Philox4x32 (PPS_PHILOX_ROUNDS rounds) on counter (x0..x3), key (k0, k1)
__device__ __forceinline__ uint4 philox(uint32_t x0, uint32_t x1, uint32_t x2, uint32_t x3, uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int r = 0; r < PPS_PHILOX_ROUNDS; ++r) {
        if (r) {
            k0 += kPhiloxW0;
            k1 += kPhiloxW1;
        }
        uint32_t hi0, lo0, hi1, lo1;
        mulhilo(kPhiloxM0, x0, hi0, lo0);
        mulhilo(kPhiloxM1, x2, hi1, lo1);
        uint32_t y0 = hi1 ^ x1 ^ k0, y2 = hi0 ^ x3 ^ k1;
        x0 = y0;
        x1 = lo1;
        x2 = y2;
        x3 = lo0;
    }
    return make_uint4(x0, x1, x2, x3);
}

__device__ __forceinline__ uint32_t lane_of(uint4 v, uint32_t lane) {
    return lane == 0 ? v.x : lane == 1 ? v.y : lane == 2 ? v.z : v.w;
}

// word of token i, arrival j (generic path: epilogues, helpers)
__device__ __forceinline__ uint32_t word_of(uint64_t key, uint64_t ctx, uint32_t pos, int64_t i, int j) {
    uint32_t k0 = (uint32_t)key ^ ((uint32_t)(j - 1) * kPhiloxW0);
    uint4 b = philox((uint32_t)((uint64_t)i >> 2), pos, (uint32_t)ctx, (uint32_t)(ctx >> 32), k0, (uint32_t)(key >> 32));
    return lane_of(b, (uint32_t)(i & 3));
}

// word of token i (first arrival) under a key (k0, k1) that every lane of the
// warp holds: callers pass values known warp-uniform (e.g. from
// __reduce_or_sync), so the compiler keeps the key schedule in uniform registers
__device__ __forceinline__ uint32_t word_of_ukey(uint32_t k0, uint32_t k1, uint64_t ctx, uint32_t pos, int64_t i) {
    const uint4 b = philox((uint32_t)((uint64_t)i >> 2), pos, (uint32_t)ctx, (uint32_t)(ctx >> 32), k0, k1);
    return lane_of(b, (uint32_t)(i & 3));
}

// Row-specialised Philox for the streaming loop (first arrival, fixed row).
// Only counter word 0 (token >> 2) varies along a row, so the products of
// the constant words in rounds 1-2 are hoisted per row: round 1 needs one
// multiply, round 2 one multiply, rounds 3-10 the usual two.
struct RowPhilox {
    uint32_t r1_c3k;          // ctx_hi ^ key_hi                         (round 1, word 2)
    uint32_t r2_f;            // lo(M1 * ctx_lo) ^ (k0 + W0)             (round 2, word 0 xor term)
    uint32_t r2_gh;           // hi(M0 * y0) ^ (k1 + W1), y0 = hi(M1*ctx_lo) ^ pos ^ k0   (round 2, word 2)
    uint32_t r2_lo0;          // lo(M0 * y0)                             (round 2, word 3)
    uint32_t rk0[PPS_PHILOX_ROUNDS - 2], rk1[PPS_PHILOX_ROUNDS - 2];  // keys of rounds 3..

    // Called by all 32 lanes of a warp with the same row.  The warp reductions
    // (of equal values) mark the row constants as warp-uniform, so the
    // compiler keeps them and the round keys in uniform registers.
    __device__ __forceinline__ void init(uint64_t key, uint64_t ctx, uint32_t pos) {
        key = ((uint64_t)__reduce_or_sync(0xffffffffu, (uint32_t)(key >> 32)) << 32) |
              __reduce_or_sync(0xffffffffu, (uint32_t)key);
        ctx = ((uint64_t)__reduce_or_sync(0xffffffffu, (uint32_t)(ctx >> 32)) << 32) |
              __reduce_or_sync(0xffffffffu, (uint32_t)ctx);
        pos = __reduce_or_sync(0xffffffffu, pos);
        init_thread(key, ctx, pos);
    }

    // The same for a thread whose row is its own (the LM-head epilogue: one row per thread).
    __device__ __forceinline__ void init_thread(uint64_t key, uint64_t ctx, uint32_t pos) {
        const uint32_t k0 = (uint32_t)key, k1 = (uint32_t)(key >> 32);
        const uint32_t c2 = (uint32_t)ctx, c3 = (uint32_t)(ctx >> 32);
        uint32_t hi1, lo1;
        mulhilo(kPhiloxM1, c2, hi1, lo1);
        const uint32_t y0 = hi1 ^ pos ^ k0;  // round-1 word 0
        r1_c3k = c3 ^ k1;
        uint32_t hi, lo;
        mulhilo(kPhiloxM0, y0, hi, lo);
        r2_lo0 = lo;
        r2_f = lo1 ^ (k0 + kPhiloxW0);
        r2_gh = hi ^ (k1 + kPhiloxW1);
#pragma unroll
        for (int r = 0; r < PPS_PHILOX_ROUNDS - 2; ++r) {
            rk0[r] = k0 + (uint32_t)(r + 2) * kPhiloxW0;
            rk1[r] = k1 + (uint32_t)(r + 2) * kPhiloxW1;
        }
    }

    // the four words of block c0 (tokens 4*c0 .. 4*c0+3)
    __device__ __forceinline__ uint4 block(uint32_t c0) const {
        uint32_t hi0, lo0;
        mulhilo(kPhiloxM0, c0, hi0, lo0);
        // round 1: (y0, y1) constant, y2 = hi0 ^ c3 ^ k1, y3 = lo0
        const uint32_t y2 = hi0 ^ r1_c3k;
        const uint32_t y3 = lo0;
        // round 2: M0*y0 constant
        uint32_t h1, l1;
        mulhilo(kPhiloxM1, y2, h1, l1);
        uint32_t x0 = h1 ^ r2_f;
        uint32_t x1 = l1;
        uint32_t x2 = y3 ^ r2_gh;
        uint32_t x3 = r2_lo0;
#pragma unroll
        for (int r = 0; r < PPS_PHILOX_ROUNDS - 2; ++r) {
            uint32_t a0, b0, a1, b1;
            mulhilo(kPhiloxM0, x0, a0, b0);
            mulhilo(kPhiloxM1, x2, a1, b1);
            const uint32_t n0 = a1 ^ x1 ^ rk0[r], n2 = a0 ^ x3 ^ rk1[r];
            x0 = n0;
            x1 = b1;
            x2 = n2;
            x3 = b0;
        }
        return make_uint4(x0, x1, x2, x3);
    }
};

// ------------------------------------------------------------------ transforms

// y = -log2 u = E log2(e) in fp32 with two MUFU operations at most:
//   u <= 1/2:          y = -lg2(u), u rounded to fp32 (relative error 2^-24, y >= 1);
//   1/2 < u, v >= 1/16: y = -lg2(1 - v) with 1 - v = u rounded to fp32 (y >= 0.093);
//   v < 1/16:          y = v log2(e) (1 + v/2 + v^2/3 + v^3/4 + v^4/5 + v^5/6), the
//                      Taylor series of -ln(1 - v) (truncation below v^6/7 < 2^-26.8).
// The largest |log2(y32) - log2(y)| over all 2^32 words is measured by
// pps_selftest_key_error and must stay below kErrAbs.
__device__ __forceinline__ float lg2_approx(float x) {
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// The first two cases are the same expression, so both values are formed and
// one is selected (no divergent branch inside a warp).
__device__ __forceinline__ float neg_log2_u(uint32_t w) {
    const float y = -lg2_approx(fmaf((float)w, 0x1p-32f, 0x1p-33f));
    const float v = fmaf((float)(~w), 0x1p-32f, 0x1p-33f);
    float p = fmaf(v, 1.0f / 6.0f, 0.2f);
    p = fmaf(v, p, 0.25f);
    p = fmaf(v, p, 1.0f / 3.0f);
    p = fmaf(v, p, 0.5f);
    p = fmaf(v, p, 1.0f);
    return (w >= 0x80000000u && v < 0.0625f) ? v * kLog2e * p : y;
}

// x = log2(-log2 u), the word part of the fp32 key
__device__ __forceinline__ float key_x32(uint32_t w) { return lg2_approx(neg_log2_u(w)); }

// fp32 key k = x - l * c with c = log2(e) / T; NaN logits map to +inf
__device__ __forceinline__ float key32(uint32_t w, float l, float c) {
    float k = fmaf(-l, c, key_x32(w));
    return k != k ? __int_as_float(0x7f800000) : k;
}

// fp64 race key s = ln E - l / T (the paper's definition, used for near-ties)
__device__ __forceinline__ double exp1_f64(uint32_t w) {
    if (w < 0x80000000u) return -log(((double)w + 0.5) * 0x1p-32);
    return -log1p(-(((double)(~w) + 0.5) * 0x1p-32));
}
__device__ __forceinline__ double key64(uint32_t w, float l, float T) {
    double ld = (double)l;
    if (ld != ld) return __longlong_as_double(0x7ff0000000000000ll);
    return log(exp1_f64(w)) - ld / (double)T;
}

// ------------------------------------------------------------------ augmented source
//
// Non-identical proposals (App. A, heterogeneous proposals): proposal b of B
// races over block b of the augmented vocabulary V x [B], the target over all
// of it with P(i)/B.  The B first arrivals of token i are generated by
// competing exponentials (the least of B iid Exp(1) is Exp(B), lies in a
// uniform block independent of its value, and the others exceed it by iid
// Exp(1) amounts):
//     E_(i,b) = E'_i / B                 in block J_i = floor(B wJ / 2^32),
//     E_(i,b) = E'_i / B + F_(i,b)       in the other blocks,
// with E'_i the token's first arrival (its word under the key), wJ its word
// under key ^ kBlockJ and F_(i,b) = Exp(1) from its word under
// key ^ (b + 1) kBlockF.  The target's augmented argmin is therefore the
// plain race on P, and a proposal's key is at least the plain key - log2 B.
constexpr uint64_t kBlockJ = 0x3C6EF372FE94F82Bull;
constexpr uint64_t kBlockF = 0xBB67AE8584CAA73Bull;

// Extra error of the fp32 block key below over the plain key's bound: the
// key is lg2.approx(fl(y' / B) [+ y_F]) - l c with y = -log2 u from
// neg_log2_u.  With M = the bound on |key_x32(w) - log2(-log2 u)| (kErrAbs,
// measured over all words) and e the absolute error of lg2.approx (at most
// 2^-17 over every fp32 input of the key's range [2^-40, 2^7), measured by
// pps_selftest_lg2_error: about 4.0e-6), each y has relative error
// <= (M + e) ln 2, the scaling and the sum add three roundings, and the outer
// lg2.approx adds e: |error| <= M + 2e + 3 * 2^-24 / ln 2 < 1.9e-5.
constexpr float kBlkErr = 4.0e-5f;

struct Blk {
    int b = 0;  // the row's block (its proposal)
    int B = 1;  // number of blocks (1: the plain race)
    // the filter tests plain keys against theta + shift, shift = ceil(log2 B) >= log2 B
    __device__ __forceinline__ float shift() const { return (float)(32 - __clz(B - 1)); }
    __device__ __forceinline__ float invB() const { return 1.0f / (float)B; }
};

__device__ __forceinline__ int block_j(uint32_t wj, int B) { return (int)__umulhi(wj, (uint32_t)B); }

// J_i and, when J_i != b, the word of the excess F_(i,b)
__device__ __forceinline__ int block_words(uint64_t key, uint64_t ctx, uint32_t pos, int64_t i, int b, int B,
                                           uint32_t& wf) {
    const int J = block_j(word_of(key ^ kBlockJ, ctx, pos, i, 1), B);
    wf = J != b ? word_of(key ^ ((uint64_t)(uint32_t)(b + 1) * kBlockF), ctx, pos, i, 1) : 0u;
    return J;
}

// the fp32 list key of block arrival E_(i,b) (key32's units: log2 E + log2 log2 e
// - l c), within key_err_bound + kBlkErr of the exact value; NaN logits -> +inf
__device__ __forceinline__ float block_key32(uint32_t w, int J, uint32_t wf, int b, float invB, float l, float c) {
    float y = neg_log2_u(w) * invB;
    if (J != b) y += neg_log2_u(wf);
    const float k = fmaf(-l, c, lg2_approx(y));
    return k != k ? __int_as_float(0x7f800000) : k;
}

// the fp64 race key s = ln E_(i,b) - l/T (near ties)
__device__ __forceinline__ double block_key64(uint32_t w, int J, uint32_t wf, int b, int B, float l, float T) {
    const double ld = (double)l;
    if (ld != ld) return __longlong_as_double(0x7ff0000000000000ll);
    double e = exp1_f64(w) / (double)B;
    if (J != b) e += exp1_f64(wf);
    return log(e) - ld / (double)T;
}

// list key of token i of a block row (words regenerated; out of line: rare path)
static __device__ __noinline__ float block_key_of(uint64_t key, uint64_t ctx, uint32_t pos, int64_t i, uint32_t w,
                                                  float l, float c, int b, int B, float invB) {
    uint32_t wf;
    const int J = block_words(key, ctx, pos, i, b, B, wf);
    return block_key32(w, J, wf, b, invB, l, c);
}

// Aaronson score A = -ln(1 - u) (Eq. 2) in fp64, and in fp32 through the key
// transform: 1 - u = (~w + 1/2) 2^-32 is the uniform of the complementary word,
// so A = ln 2 * neg_log2_u(~w).  The transform's relative error is below
// 2^kErrAbs - 1 < 2.1e-6 for every word (pps_selftest_key_error checks all
// 2^32), 2.2e-6 with the final product; its absolute error is below 2e-7.
__device__ __forceinline__ double score64(uint32_t w) {
    if (w < 0x80000000u) return -log1p(-(((double)w + 0.5) * 0x1p-32));
    return -log(((double)(~w) + 0.5) * 0x1p-32);
}
__device__ __forceinline__ float score32(uint32_t w) { return 0.69314718055994531f * neg_log2_u(~w); }

// Detection score kinds of the pivot r = u (App. D): Aaronson -ln(1 - r), the
// U-score r, Li et al.'s h*_{gum,Delta}(r) = ln(k r^a + [q > 0] r^b) with
// a = Delta/(1-Delta), b = (1-q)/q, and the truncated power law
// min(cap, (1-r)^(-1/2)) - centre.  Constants come from the host.
__device__ __forceinline__ float score_kind32(uint32_t w, const ScoreParams& P) {
    if (P.kind == 0) return score32(w);
    const float u = fmaf((float)w, 0x1p-32f, 0x1p-33f);     // r
    const float v = fmaf((float)(~w), 0x1p-32f, 0x1p-33f);  // 1 - r
    if (P.kind == 1) return w < 0x80000000u ? u : 1.0f - v;
    if (P.kind == 2) {
        const float lr = w < 0x80000000u ? logf(u) : log1pf(-v);
        const float x = P.k * expf(P.a * lr) + (P.has_q != 0.0f ? expf(P.b * lr) : 0.0f);
        return logf(x);
    }
    return fminf(P.cap, 1.0f / sqrtf(v)) - P.centre;
}

// fp32 key k = log2(E) + log2(log2 e) - l log2(e)/T  ->  s = ln E - l/T = (k - log2(log2 e)) ln 2
__device__ __forceinline__ float key_to_s(float k) { return (k + kLog2Ln2) * 0.69314718055994530942f; }

// ------------------------------------------------------------------ filter
//
// A token can enter a list only if its fp32 key is below theta.  Since
// E = -ln(1 - v) >= v with v = 1 - u = (~w + 1/2) 2^-32, a key below theta
// needs v < e_z := 2^(theta + l c) ln 2, i.e. (with a = (~w) >> 9, so that
// ~w >= 512 a) a < T := e_z 2^23.  With b = w >> 9, a = 2^23 - 1 - b, so the
// token can be dropped when T + 2^23 + b <= 2^24 - 1.  The sum is formed in
// fp32 from the bit pattern 0x4b000000 + b (= 2^23 + b exactly, one mad.hi
// on the multiply pipe) plus T; its rounding error is below 1, so testing
// S >= 2^24 - 2 never drops a token that could enter.  tz carries
// theta + margin + log2(ln 2) + 23 (+inf while the list is not full); NaN
// logits give S = NaN and are dropped.
__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
#ifndef PPS_FILTER
#define PPS_FILTER 0
#endif
#if PPS_FILTER == 0
// 2^23 + (w >> 9) as fp32 bits from one mad.hi; cut 2^24 - 2, T scaled by 2^23
constexpr float kFilterScaleLog2 = 23.0f;
constexpr float kFilterCut = 16777214.0f;  // 2^24 - 2
__device__ __forceinline__ float filter_word(uint32_t w) {
    uint32_t bb;
    asm("mad.hi.u32 %0, %1, %2, %3;" : "=r"(bb) : "r"(w), "r"(1u << 23), "r"(0x4b000000u));
    return __uint_as_float(bb);
}
#else
// 0x4b000000 | (w >> 8) as fp32 bits from one byte permute: 2^23 + (w >> 8) for
// w < 2^31 and 2 (w >> 8) above; the token can be dropped when T + f <= 2^25 - 2
// (T scaled by 2^25), and the fp32 sum errs by at most 2, so the cut is 2^25 - 4.
// Below 2^31 the test drops only words with u < 3/4 - e_z, inside the safe
// region u <= 1 - e_z.
constexpr float kFilterScaleLog2 = 25.0f;
constexpr float kFilterCut = 33554428.0f;  // 2^25 - 4
__device__ __forceinline__ float filter_word(uint32_t w) { return __uint_as_float(__byte_perm(w, 0x4bu, 0x4321)); }
#endif
__device__ __forceinline__ float filter_sum(uint32_t w, float l, float c, float tz) {
    return ex2_approx(fmaf(l, c, tz)) + filter_word(w);
}
__device__ __forceinline__ bool filter_pass(uint32_t w, float l, float c, float tz) {
    return filter_sum(w, l, c, tz) >= kFilterCut;
}
__device__ __forceinline__ float filter_tz(float theta) {
    return theta + (kFilterMargin + kLog2Ln2 + kFilterScaleLog2);
}

// packed bf16 max (a NaN half yields the other operand's half)
__device__ __forceinline__ uint32_t bf2_max(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("max.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}

// bf16 -> fp32 (exact)
__device__ __forceinline__ float bf16_lo(uint32_t x) { return __uint_as_float(x << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t x) { return __uint_as_float(x & 0xffff0000u); }

}  // namespace pps
