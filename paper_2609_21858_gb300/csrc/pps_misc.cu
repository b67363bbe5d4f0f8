// pps_misc.cu -- detector pass, raw keyed words, and the fp32 key self-test.
#include <climits>
#include <cstdint>

#include "pps_device.cuh"
#include "pps_internal.h"

namespace pps {

#define FULL 0xffffffffu

// Detector (App. E): every warp takes a contiguous chunk of tokens and works
// through it a group of 128 at a time; lane l loads and scores tokens
// 4l .. 4l+3 of the group (16-byte loads when the arrays are aligned).  When
// the whole group has one key (the tokens of one text), the Philox key
// schedule is warp-uniform and kept in uniform registers.  Segment sums: when a
// group lies inside the open segment (segments of a text are usually longer
// than a group), each lane adds its four scores and one warp reduction adds
// the group to the segment's running sum; a group that holds a segment
// boundary is rearranged to lane-major order (shuffles) and takes a segmented
// warp scan per 32 tokens.  The running sum is a
// float-float pair (an exact fp32 two-sum per addition, FP64 being slow on this
// part) and goes to the segment's fp64 slot with one atomic per segment end the
// warp sees (plus one at the end of its chunk).
constexpr int kScoreAhead = 4;  // iterations whose inputs a warp loads together


// hi + lo += v, with the rounding error of hi + v kept in lo (two-sum)
__device__ __forceinline__ void ff_add(float& hi, float& lo, float v) {
    const float s = hi + v;
    const float bp = s - hi;
    lo += (hi - (s - bp)) + (v - bp);
    hi = s;
}

template <bool VEC>
__global__ void __launch_bounds__(256) wm_score_kernel(const int32_t* __restrict__ tokens,
                                                       const uint64_t* __restrict__ key,
                                                       const uint64_t* __restrict__ ctx,
                                                       const uint32_t* __restrict__ pos, int64_t n, int32_t n_seg,
                                                       const int64_t* __restrict__ seg_off, ScoreParams P,
                                                       float* out_score, double* out_sum, int64_t chunk) {
    const int lane = threadIdx.x & 31;
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t c0 = gw * chunk;
    if (c0 >= n) return;
    const int64_t c1 = min(n, c0 + chunk);
    const bool segs = out_sum != nullptr && seg_off != nullptr;
    // the open segment (warp-uniform): the segment of the chunk's first token (binary search, lane 0)
    int seg = 0;
    int64_t seg_end = LLONG_MAX;
    if (segs) {
        if (lane == 0) {
            int lo = 0, hi = n_seg;  // seg_off[lo] <= c0 < seg_off[hi]
            while (hi - lo > 1) {
                int mid = (lo + hi) >> 1;
                if (seg_off[mid] <= c0)
                    lo = mid;
                else
                    hi = mid;
            }
            seg = lo;
        }
        seg = __shfl_sync(FULL, seg, 0);
        seg_end = seg + 1 < n_seg ? seg_off[seg + 1] : LLONG_MAX;
    }
    float chi = 0.0f, clo = 0.0f;  // running sum of the open segment
    constexpr int G = 32 * kScoreAhead;
    static_assert(kScoreAhead == 4, "a lane holds four consecutive tuples of a group");
    for (int64_t grp = c0; grp < c1; grp += G) {
        // lane l holds tuples grp + 4 l .. grp + 4 l + 3 (the first nloc of them exist), loaded
        // with 16-byte loads when the arrays allow it
        const int64_t t0 = grp + 4 * lane;
        const int nloc = (int)max((int64_t)0, min((int64_t)4, c1 - t0));
        int32_t tk[4] = {0, 0, 0, 0};
        uint64_t kk[4] = {0, 0, 0, 0}, cx[4] = {0, 0, 0, 0};
        uint32_t ps[4] = {0, 0, 0, 0};
        if (VEC && nloc == 4) {
            const int4 t4 = __ldg(reinterpret_cast<const int4*>(tokens + t0));
            const uint4 p4 = __ldg(reinterpret_cast<const uint4*>(pos + t0));
            const ulonglong2 ka = __ldg(reinterpret_cast<const ulonglong2*>(key + t0));
            const ulonglong2 kb = __ldg(reinterpret_cast<const ulonglong2*>(key + t0 + 2));
            const ulonglong2 xa = __ldg(reinterpret_cast<const ulonglong2*>(ctx + t0));
            const ulonglong2 xb = __ldg(reinterpret_cast<const ulonglong2*>(ctx + t0 + 2));
            tk[0] = t4.x; tk[1] = t4.y; tk[2] = t4.z; tk[3] = t4.w;
            ps[0] = p4.x; ps[1] = p4.y; ps[2] = p4.z; ps[3] = p4.w;
            kk[0] = ka.x; kk[1] = ka.y; kk[2] = kb.x; kk[3] = kb.y;
            cx[0] = xa.x; cx[1] = xa.y; cx[2] = xb.x; cx[3] = xb.y;
        } else {
#pragma unroll
            for (int u = 0; u < 4; ++u)
                if (u < nloc) {
                    tk[u] = tokens[t0 + u];
                    ps[u] = pos[t0 + u];
                    kk[u] = key[t0 + u];
                    cx[u] = ctx[t0 + u];
                }
        }
        // one key for the whole group (the tokens of one text): its schedule in uniform registers
        bool same = true;
#pragma unroll
        for (int u = 1; u < 4; ++u) same &= u >= nloc || kk[u] == kk[0];
        const uint64_t k_any = nloc > 0 ? kk[0] : 0ull;
        const uint32_t klo = __reduce_or_sync(FULL, (uint32_t)k_any), khi = __reduce_or_sync(FULL, (uint32_t)(k_any >> 32));
        same &= nloc == 0 || k_any == (((uint64_t)khi << 32) | klo);
        const bool ukey = __all_sync(FULL, same);
        float A[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            A[u] = 0.0f;
            if (u < nloc) {
                const uint32_t w = ukey ? word_of_ukey(klo, khi, cx[u], ps[u], (int64_t)tk[u])
                                        : word_of(kk[u], cx[u], ps[u], (int64_t)tk[u], 1);
                A[u] = score_kind32(w, P);
            }
        }
        if (out_score) {
            if (VEC && nloc == 4)
                *reinterpret_cast<float4*>(out_score + t0) = make_float4(A[0], A[1], A[2], A[3]);
            else
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (u < nloc) out_score[t0 + u] = A[u];
        }
        if (!out_sum) continue;
        const int64_t gend = min(grp + 32 * kScoreAhead, c1);
        if (segs && grp >= seg_end) {
            // the open segment ended before this group: flush it, move to the group's first segment
            if (lane == 0 && (chi != 0.0f || clo != 0.0f)) atomicAdd(out_sum + seg, (double)chi + (double)clo);
            chi = clo = 0.0f;
            do {
                ++seg;
            } while (seg + 1 < n_seg && seg_off[seg + 1] <= grp);
            seg_end = seg + 1 < n_seg ? seg_off[seg + 1] : LLONG_MAX;
        }
        if (gend <= seg_end) {
            // the whole group lies in the open segment (or there is one segment)
            float v = A[0];
#pragma unroll
            for (int u = 1; u < kScoreAhead; ++u) v += A[u];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL, v, o);
            ff_add(chi, clo, v);
            continue;
        }
        // a segment boundary inside the group: a segmented scan per iteration, over the
        // lane-major layout (iteration u, lane t: tuple grp + 32 u + t, held by lane 8 u + t / 4)
        float Am[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int src = 8 * u + (lane >> 2);
            const float a0 = __shfl_sync(FULL, A[0], src), a1 = __shfl_sync(FULL, A[1], src);
            const float a2 = __shfl_sync(FULL, A[2], src), a3 = __shfl_sync(FULL, A[3], src);
            const int e = lane & 3;
            Am[u] = e == 0 ? a0 : e == 1 ? a1 : e == 2 ? a2 : a3;
        }
#pragma unroll
        for (int u = 0; u < kScoreAhead; ++u) {
            const int64_t base = grp + 32 * u;
            if (base >= c1) break;
            const int64_t t = base + lane;
            // segment of my token, advanced from the warp's open segment (segments are contiguous)
            int my = INT_MAX;
            if (t < c1) {
                my = seg;
                while (my + 1 < n_seg && seg_off[my + 1] <= t) ++my;
            }
            // segmented inclusive scan over the lanes of each segment run
            float v = Am[u];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const float ov = __shfl_up_sync(FULL, v, o);
                const int os = __shfl_up_sync(FULL, my, o);
                if (lane >= o && os == my) v += ov;
            }
            // the open segment ended before this iteration's first run: flush it
            const int s0 = __shfl_sync(FULL, my, 0);
            if (s0 != seg) {
                if (lane == 0 && (chi != 0.0f || clo != 0.0f)) atomicAdd(out_sum + seg, (double)chi + (double)clo);
                chi = clo = 0.0f;
                seg = s0;
            }
            const int nxt = __shfl_down_sync(FULL, my, 1);
            const bool more = base + 32 < c1;
            if (t < c1 && (lane == 31 || nxt != my)) {
                const bool open = lane == 31 && more;  // may continue into the next iteration
                if (!open) atomicAdd(out_sum + my, (double)v + (my == seg ? (double)chi + (double)clo : 0.0));
            }
            if (more) {
                const float v31 = __shfl_sync(FULL, v, 31);
                const int s31 = __shfl_sync(FULL, my, 31);
                if (s31 == seg) {
                    ff_add(chi, clo, v31);
                } else {
                    chi = v31;
                    clo = 0.0f;
                }
                seg = s31;
            } else {
                chi = clo = 0.0f;
            }
        }
        seg_end = seg + 1 < n_seg ? seg_off[seg + 1] : LLONG_MAX;
    }
    // the chunk's open sum (the scan path flushes its own at the chunk's end)
    if (out_sum && lane == 0 && (chi != 0.0f || clo != 0.0f))
        atomicAdd(out_sum + (segs ? seg : 0), (double)chi + (double)clo);
}

// ln Gamma(x) for x >= 16 by Stirling's asymptotic series (truncation error
// below 1e-16 there); smaller x through the recurrence Gamma(x+1) = x Gamma(x).
__device__ double lgamma_stirling(double x) {
    double shift = 0.0;
    while (x < 16.0) {
        shift -= log(x);
        x += 1.0;
    }
    const double r = 1.0 / x, r2 = r * r;
    const double series = r * (1.0 / 12.0 - r2 * (1.0 / 360.0 - r2 * (1.0 / 1260.0 - r2 * (1.0 / 1680.0))));
    return shift + (x - 0.5) * log(x) - x + 0.91893853320467274178 + series;
}

// Stirling's series of ln Gamma(M) - (M - 1/2) ln M + M - ln sqrt(2 pi) for M >= 16
// (1/(12M) and its next three terms; below 1e-3 there, so fp32 suffices)
__device__ __forceinline__ float stirling_tail(float M) {
    const float r = 1.0f / M, r2 = r * r;
    return r * (1.0f / 12.0f - r2 * (1.0f / 360.0f - r2 * (1.0f / 1260.0f - r2 * (1.0f / 1680.0f))));
}

// ln of the Poisson term e^-S S^k / k! for k = M - 1 (top = false) or k = M (top = true).
// For M >= 16, with y = S/M - 1 and Stirling's formula for ln Gamma(M) (ln M! = ln Gamma(M)
// + ln M), both are k log1p(y) - (S - M) - ln sqrt(2 pi M) - stirling_tail(M): the large
// parts S and k ln S cancel against M and k ln M inside log1p, so one fp64 log1p is the
// only fp64 transcendental, and the M-only terms (below ~12) are fp32 (errors < 1e-6).
// Smaller M take ln Gamma from lgamma_stirling.
__device__ double poisson_lead(int64_t M, double S, bool top) {
    if (M < 16) {
        const double ls = log(S);
        return top ? -S + (double)M * ls - lgamma_stirling((double)M + 1.0)
                   : -S + (double)(M - 1) * ls - lgamma_stirling((double)M);
    }
    const double Md = (double)M;
    double rM = (double)(1.0f / (float)M);
    rM = rM * (2.0 - Md * rM);  // one Newton step: relative error ~1e-14
    const double y = (S - Md) * rM;
    const float Mf = (float)M;
    const float c = 0.5f * logf(6.28318530717958648f * Mf) + stirling_tail(Mf);
    return (top ? Md : Md - 1.0) * log1p(y) - (S - Md) - (double)c;
}

// The ratios r_m (r_0 = 1) of the Poisson terms to the leading one, summed in
// compensated (Kahan) fp32 until a term drops below 1e-12 of the sum: downward
// (S >= M: r_m = r_{m-1} (M - m) / S, s = 1/S in fp32) or upward (S < M:
// r_m = r_{m-1} S / (M + m), s = S in fp32).  Also returns sum_m m r_m, the
// first-order sensitivity to the relative error of s.  For M < kSeriesF64Min,
// where the counters are exact in fp32 (int64 -> fp32 conversions in the loop
// cost a quarter of the kernel).
template <bool DOWN>
__device__ __forceinline__ void poisson_ratios(int64_t M, float s, float& sum, float& wsum) {
    float r = 1.0f, comp = 0.0f, m = 0.0f;
    sum = 1.0f;
    wsum = 0.0f;
    for (float j = (float)(DOWN ? M - 1 : M + 1); !DOWN || j > 0.0f; j += DOWN ? -1.0f : 1.0f) {
        r *= DOWN ? j * s : s / j;
        m += 1.0f;
        const float y = r - comp, t = sum + y;
        comp = (t - sum) - y;
        sum = t;
        wsum = fmaf(m, r, wsum);
        if (r < 1e-12f * sum) break;
    }
}

// From this segment length on the series runs in fp64: with S near M, successive
// ratios j/S differ by ~1/M, below the fp32 spacing near 1 for M ~ 2^24, so their
// rounding errors stop averaging out and the fp32 product drifts (measured on the
// host: 7e-7 in ln p at M = 2^16, 1.3e-5 at 2^24).  Such segments are rare; their
// ~6 sqrt(M) fp64 steps cost microseconds.
constexpr int64_t kSeriesF64Min = 1 << 18;

// ln P(Gamma(M,1) >= S) for integer M >= 1, as the Poisson probability
// P(N <= M-1), N ~ Poisson(S).  The leading term e^-S S^j / j! at j = M-1
// (S >= M) or j = M (S < M) is taken in fp64 (poisson_lead); the sum of the
// ratios of the other terms to it, all <= 1 and summed away from the mode
// until they stop mattering: for S >= M downward from M-1 (ratios j/S), below
// as 1 - P(N >= M) upward from M (ratios S/j).  Below kSeriesF64Min tokens in
// compensated fp32 (poisson_ratios; FP64 throughput is low on this part) with a
// first-order correction for the fp32 image of S (the m-th term carries it m
// times: with its relative error d, the exact sum is sum + d * sum_m m r_m);
// error below 1e-6 absolute in ln p.  From kSeriesF64Min on in fp64.
__device__ double gamma_tail_logp(int64_t M, double S) {
    if (!(S > 0.0)) return 0.0;
    if (M >= kSeriesF64Min) {
        double r = 1.0, sum = 1.0;
        if (S >= (double)M) {
            const double inv = 1.0 / S;
            for (int64_t j = M - 1; j > 0; --j) {
                r *= (double)j * inv;
                sum += r;
                if (r < 1e-17 * sum) break;
            }
            return poisson_lead(M, S, false) + log(sum);
        }
        for (int64_t j = M + 1;; ++j) {
            r *= S / (double)j;
            sum += r;
            if (r < 1e-17 * sum) break;
        }
        return log1p(-exp(poisson_lead(M, S, true)) * sum);
    }
    const float Sf = (float)S;
    float sum, wsum;
    if (S >= (double)M) {
        const float inv = 1.0f / Sf;
        // d = (1/S) / inv - 1 = e / (1 - e) with e = 1 - S inv (|e| < 1e-7): e + e^2
        const double e = 1.0 - S * (double)inv;
        const double d = fma(e, e, e);
        poisson_ratios<true>(M, inv, sum, wsum);
        // tot in [1, ~1e3]: its logarithm in fp32 errs by ~1e-7 absolute
        const double tot = (double)sum + d * (double)wsum;
        return poisson_lead(M, S, false) + (double)logf((float)tot);
    }
    const double d = (S - (double)Sf) * (double)(1.0f / Sf);  // relative error of Sf (its own error ~1e-14)
    poisson_ratios<false>(M, Sf, sum, wsum);
    // S < M: P(N >= M) <= ~1/2, so ln(1 - P(N >= M)) in fp32 errs by ~1e-7 absolute
    const double tot = (double)sum + d * (double)wsum;
    const double lead = poisson_lead(M, S, true);
    return (double)log1pf(-expf((float)lead) * (float)tot);
}

// Chernoff bound on ln P(U_1 + ... + U_M >= S): the exponent
// M ln((e^l - 1)/l) - l S at the l where the mean of the exponentially tilted
// uniform, 1/(1 - e^-l) - 1/l, equals S/M (fp32 Newton steps kept inside a
// bisection bracket; the exponent is flat there, and is evaluated in fp64).
// 0 for S <= M/2, -inf for S >= M.
__device__ double chernoff_u_logp(int64_t M, double S) {
    const double x = S / (double)M;
    if (!(x > 0.5)) return 0.0;
    if (x >= 1.0) return -INFINITY;
    const float xf = (float)x;
    auto mean = [](float l) {
        if (l < 1e-2f) return 0.5f + l / 12.0f - l * l * l / 720.0f;
        return 1.0f / (-expm1f(-l)) - 1.0f / l;
    };
    auto slope = [](float l) {  // variance of the tilted uniform
        if (l < 1e-2f) return 1.0f / 12.0f - l * l / 240.0f;
        const float e = expf(-l), d = -expm1f(-l);
        return 1.0f / (l * l) - e / (d * d);
    };
    float lo = 0.0f, hi = 2.0f / (1.0f - xf) + 10.0f;
    float l = xf < 0.75f ? 12.0f * (xf - 0.5f) : 1.0f / (1.0f - xf);
    for (int it = 0; it < 60; ++it) {
        const float f = mean(l) - xf;
        if (f > 0.0f) hi = l;
        else lo = l;
        float nl = l - f / slope(l);
        if (!(nl > lo && nl < hi)) nl = 0.5f * (lo + hi);
        if (fabsf(nl - l) <= 1e-6f * l) {
            l = nl;
            break;
        }
        l = nl;
    }
    const double ld = (double)l;
    const double e = (double)M * log(expm1(ld) / ld) - ld * S;
    return e < 0.0 ? e : 0.0;
}

// per-segment ln p-values from the segment sums (kind 0 Gamma tail, 1 Chernoff on U)
__global__ void seg_logp_kernel(int64_t n, int32_t n_seg, const int64_t* __restrict__ seg_off,
                                const double* __restrict__ sums, int kind, double* out_logp) {
    const int g = blockIdx.x * blockDim.x + threadIdx.x;
    if (g >= n_seg) return;
    const int64_t M = seg_off ? seg_off[g + 1] - seg_off[g] : n;
    double lp;
    if (M <= 0)
        lp = 0.0;
    else if (kind == 0)
        lp = gamma_tail_logp(M, sums[g]);
    else if (kind == 1)
        lp = chernoff_u_logp(M, sums[g]);
    else
        lp = __longlong_as_double(0x7ff8000000000000ll);  // NaN: no null law for this score
    out_logp[g] = lp;
}

// SplitMix64's output function (Steele, Lea, Flood, OOPSLA'14): the labeler of
// a child context, label(c || u) = mix(label(c) ^ (u + 1) * 0x9E3779B97F4A7C15)
__device__ __forceinline__ uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

// One depth of the dynamic IID draft tree (layout in pps.h): warp b takes
// sequence b, lane i the depth's row i; the distinct labels of the present
// rows get consecutive child slots (exclusive scan over the rows).
__global__ void tree_expand_kernel(int32_t n_seq, int32_t K, int32_t gamma, int32_t depth,
                                   const int32_t* __restrict__ tok, const int32_t* __restrict__ mult,
                                   const int32_t* __restrict__ ndist, const uint64_t* __restrict__ key,
                                   const uint64_t* __restrict__ ctx, const uint32_t* __restrict__ pos,
                                   const int32_t* __restrict__ row_k, uint64_t* next_key, uint64_t* next_ctx,
                                   uint32_t* next_pos, int32_t* next_k, int32_t* child_node, uint64_t* node_key,
                                   uint64_t* node_ctx, uint32_t* node_pos) {
    pdl_wait();  // the lists and row ids of the previous launch
    pdl_launch_dependents();
    const int lane = threadIdx.x & 31;
    const int64_t b = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (b >= n_seq) return;
    const int64_t N1 = 1 + (int64_t)K * gamma;
    const int w = depth == 0 ? 1 : K;
    // draft rows are numbered depth-major: depth d's rows start at D_d = n_seq (1 + (d-1) K)
    const int64_t D_d = depth == 0 ? 0 : (int64_t)n_seq * (1 + (int64_t)(depth - 1) * K), off_n = 1 + (int64_t)depth * K;
    const int64_t r = b * w + lane;
    const bool row = lane < w;
    int nd = 0;
    if (row && row_k[r] > 0) nd = max(0, min(ndist[r], K));
    int j0 = nd;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(FULL, j0, o);
        if (lane >= o) j0 += t;
    }
    const int total = min(__shfl_sync(FULL, j0, 31), K);
    j0 -= nd;
    if (row) {
        const int64_t dr = D_d + b * w + lane;
        for (int m = 0; m < K; ++m) {
            int node = -1;
            const int j = j0 + m;
            if (m < nd && j < K) {
                const int64_t q = b * K + j;
                const uint64_t lab = mix64(ctx[r] ^ ((uint64_t)(uint32_t)(tok[r * K + m] + 1) * 0x9E3779B97F4A7C15ull));
                next_key[q] = key[r];
                next_ctx[q] = lab;
                next_pos[q] = pos[r] + 1u;
                next_k[q] = mult[r * K + m];
                node = (int)(b * N1 + off_n + j);
                node_key[node] = key[r];
                node_ctx[node] = lab;
                node_pos[node] = pos[r] + 1u;
            }
            child_node[dr * K + m] = node;
        }
    }
    for (int j = lane; j < K; j += 32)
        if (j >= total) {
            const int64_t q = b * K + j;
            next_key[q] = key[b * w];
            next_ctx[q] = 0;
            next_pos[q] = 0;
            next_k[q] = 0;
        }
}

// One depth of the draft tree of B non-identical proposals (layout in pps.h):
// warp s takes sequence s, lane b proposal b.  A proposal at node o of depth
// d that drew token x moves to child (d+1, f), f = the first proposal at the
// same node that drew x; node o's list holds the distinct tokens of its
// proposals in proposal order, each with that child.
__global__ void hetero_expand_kernel(int32_t n_seq, int32_t B, int32_t gamma, int32_t depth,
                                     const int32_t* __restrict__ tok, const uint64_t* __restrict__ key,
                                     const uint64_t* __restrict__ ctx, const uint32_t* __restrict__ pos,
                                     const int32_t* __restrict__ owner, uint64_t* next_key, uint64_t* next_ctx,
                                     uint32_t* next_pos, int32_t* next_owner, int32_t* list_tok, int32_t* list_nd,
                                     int32_t* child_node, uint64_t* node_key, uint64_t* node_ctx,
                                     uint32_t* node_pos) {
    pdl_wait();  // the lists and row ids of the previous launch
    pdl_launch_dependents();
    const int lane = threadIdx.x & 31;
    const int64_t s = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (s >= n_seq) return;
    const int64_t N1 = 1 + (int64_t)B * gamma;
    const int w = depth == 0 ? 1 : B;
    // node lists are numbered depth-major: depth d's start at L_d = n_seq (1 + (d-1) B)
    const int64_t L_d = depth == 0 ? 0 : (int64_t)n_seq * (1 + (int64_t)(depth - 1) * B);
    const int64_t child0 = s * N1 + 1 + (int64_t)depth * B;  // node (s, d+1, 0)
    const int64_t r = s * B + lane;
    int o = -1, x = -1;
    if (lane < B) {
        o = owner[r];
        x = tok[r];
    }
    const bool alive = lane < B && o >= 0 && o < w && x >= 0;
    int first = alive ? lane : -1;
    for (int t = 0; t < B; ++t) {
        const int ot = __shfl_sync(FULL, o, t), xt = __shfl_sync(FULL, x, t);
        const bool at = __shfl_sync(FULL, (int)alive, t) != 0;
        if (alive && at && t < first && ot == o && xt == x) first = t;
    }
    // lane o writes the list of node (s, d, o)
    const int64_t lr = L_d + s * w + lane;
    int m = 0;
    for (int t = 0; t < B; ++t) {
        const int ot = __shfl_sync(FULL, o, t), xt = __shfl_sync(FULL, x, t), ft = __shfl_sync(FULL, first, t);
        const bool at = __shfl_sync(FULL, (int)alive, t) != 0;
        if (lane < w && at && ot == lane && ft == t) {
            list_tok[lr * B + m] = xt;
            child_node[lr * B + m] = (int32_t)(child0 + t);
            ++m;
        }
    }
    if (lane < w) {
        for (int q = m; q < B; ++q) {
            list_tok[lr * B + q] = -1;
            child_node[lr * B + q] = -1;
        }
        list_nd[lr] = m;
    }
    // depth d+1: node (s, d+1, b) is proposal b's when it is the first to reach it
    if (lane < B) {
        uint64_t k = 0, lab = 0;
        uint32_t p = 0;
        if (alive) {
            k = key[r];
            lab = mix64(ctx[r] ^ ((uint64_t)(uint32_t)(x + 1) * 0x9E3779B97F4A7C15ull));
            p = pos[r] + 1u;
        }
        const bool owns = alive && first == lane;
        node_key[child0 + lane] = owns ? k : 0;
        node_ctx[child0 + lane] = owns ? lab : 0;
        node_pos[child0 + lane] = owns ? p : 0u;
        if (depth + 1 < gamma) {
            next_key[r] = k;
            next_ctx[r] = lab;
            next_pos[r] = p;
            next_owner[r] = alive ? first : -1;
        }
    }
}

// block J of the augmented race's winning point (Y, J) for each token
__global__ void hetero_block_kernel(int64_t n, int32_t B, const int32_t* __restrict__ tok,
                                    const uint64_t* __restrict__ key, const uint64_t* __restrict__ ctx,
                                    const uint32_t* __restrict__ pos, int32_t* __restrict__ out) {
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < n; t += (int64_t)gridDim.x * blockDim.x) {
        const int32_t y = tok[t];
        out[t] = y >= 0 ? block_j(word_of(key[t] ^ kBlockJ, ctx[t], pos[t], y, 1), B) : -1;
    }
}

__global__ void words_kernel(const uint64_t* __restrict__ key, const uint64_t* __restrict__ ctx,
                             const uint32_t* __restrict__ pos, int64_t n_rows, int64_t V, int32_t arrival,
                             uint32_t* __restrict__ out) {
    const int64_t total = n_rows * V;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total; t += (int64_t)gridDim.x * blockDim.x) {
        int64_t r = t / V, i = t - r * V;
        out[t] = word_of(key[r], ctx[r], pos[r], i, arrival);
    }
}

// largest |x32(w) - log2(-log2 u(w))| over a word range; the fp64 reference
// uses E = -ln u through u for u <= 1/2 and through v = 1 - u above
__global__ void selftest_kernel(uint64_t w0, uint64_t w1, float* out) {
    float worst = 0.0f;
    for (uint64_t w = w0 + (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; w < w1;
         w += (uint64_t)gridDim.x * blockDim.x) {
        uint32_t x = (uint32_t)w;
        float x32 = key_x32(x);
        double xd = log2(exp1_f64(x) * 1.4426950408889634074);
        float d = (float)fabs((double)x32 - xd);
        worst = fmaxf(worst, d);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) worst = fmaxf(worst, __shfl_xor_sync(FULL, worst, o));
    if ((threadIdx.x & 31) == 0) atomicMax(reinterpret_cast<unsigned int*>(out), __float_as_uint(worst));
}

// largest |lg2.approx(x) - log2 x| over the positive fp32 x with bit patterns
// in [b0, b1) (every input of the block key's outer logarithm)
__global__ void selftest_lg2_kernel(uint32_t b0, uint32_t b1, float* out) {
    float worst = 0.0f;
    for (uint64_t b = (uint64_t)b0 + (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; b < b1;
         b += (uint64_t)gridDim.x * blockDim.x) {
        const float x = __uint_as_float((uint32_t)b);
        const float d = (float)fabs((double)lg2_approx(x) - log2((double)x));
        worst = fmaxf(worst, d);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) worst = fmaxf(worst, __shfl_xor_sync(FULL, worst, o));
    if ((threadIdx.x & 31) == 0) atomicMax(reinterpret_cast<unsigned int*>(out), __float_as_uint(worst));
}

// Philox-only throughput: every thread generates blocks c0 = t, t + stride, ...
// with the row-specialised generator of the streaming kernels and folds the
// words into one value, so the kernel is bound by the Philox multiplies alone
// (the ceiling of the race kernels on bf16 rows).
__global__ void __launch_bounds__(256) philox_rate_kernel(uint64_t key, uint64_t ctx, uint32_t pos, uint64_t n_blocks,
                                                          uint32_t* out) {
    RowPhilox rp;
    rp.init(key, ctx, pos);
    uint32_t acc = 0;
    const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
    for (uint64_t b = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; b < n_blocks; b += 2 * stride) {
        const uint4 v0 = rp.block((uint32_t)b);
        const uint4 v1 = rp.block((uint32_t)(b + stride));
        acc ^= v0.x ^ v0.y ^ v0.z ^ v0.w ^ v1.x ^ v1.y ^ v1.z ^ v1.w;
    }
    out[(uint64_t)blockIdx.x * blockDim.x + threadIdx.x] = acc;
}

cudaError_t launch_philox_rate(uint64_t n_blocks, uint32_t* out, int out_len, cudaStream_t stream) {
    int blocks = out_len / 256;
    if (blocks < 1) return cudaErrorInvalidValue;
    philox_rate_kernel<<<blocks, 256, 0, stream>>>(0x0123456789abcdefull, 0xfedcba9876543210ull, 7u, n_blocks, out);
    return cudaGetLastError();
}

cudaError_t launch_wm_score(const int32_t* tokens, const uint64_t* key, const uint64_t* ctx, const uint32_t* pos,
                            int64_t n, int32_t n_seg, const int64_t* seg_off, const ScoreParams& P, float* out_score,
                            double* out_sum, double* out_logp, cudaStream_t stream) {
    const int32_t ns = seg_off ? n_seg : 1;
    if (out_sum) {
        cudaError_t e = cudaMemsetAsync(out_sum, 0, sizeof(double) * (size_t)ns, stream);
        if (e != cudaSuccess) return e;
    }
    if (n > 0) {
        // one wave: as many warps as the GPU holds at once, each a contiguous chunk
        // (a multiple of the 128 tokens of one load group)
        const int64_t resident =
            (int64_t)device_sm_count() * resident_ctas(kOccScore, (const void*)wm_score_kernel<true>, 256) * (256 / 32);
        const int64_t group = 32 * kScoreAhead;
        const int64_t chunk = ((n + resident - 1) / resident + group - 1) / group * group;
        const int64_t warps = (n + chunk - 1) / chunk;
        const int64_t blocks = (warps * 32 + 255) / 256;
        // 16-byte loads and stores need 16-byte aligned arrays (chunks start on multiples of 128 tuples)
        auto al = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
        const bool vec = al(tokens) && al(key) && al(ctx) && al(pos) && (out_score == nullptr || al(out_score));
        if (vec)
            wm_score_kernel<true><<<(unsigned)blocks, 256, 0, stream>>>(tokens, key, ctx, pos, n, n_seg, seg_off, P,
                                                                        out_score, out_sum, chunk);
        else
            wm_score_kernel<false><<<(unsigned)blocks, 256, 0, stream>>>(tokens, key, ctx, pos, n, n_seg, seg_off, P,
                                                                         out_score, out_sum, chunk);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    if (out_logp && ns > 0) {
        seg_logp_kernel<<<(ns + 127) / 128, 128, 0, stream>>>(n, ns, seg_off, out_sum, P.kind, out_logp);
        return cudaGetLastError();
    }
    return cudaSuccess;
}

cudaError_t launch_tree_expand(int32_t n_seq, int32_t K, int32_t gamma, int32_t depth, const int32_t* tok,
                               const int32_t* mult, const int32_t* ndist, const uint64_t* key, const uint64_t* ctx,
                               const uint32_t* pos, const int32_t* row_k, uint64_t* next_key, uint64_t* next_ctx,
                               uint32_t* next_pos, int32_t* next_k, int32_t* child_node, uint64_t* node_key,
                               uint64_t* node_ctx, uint32_t* node_pos, cudaStream_t stream) {
    if (n_seq == 0) return cudaSuccess;
    const int64_t blocks = ((int64_t)n_seq * 32 + 255) / 256;
    const cudaError_t e = launch_pdl(tree_expand_kernel, dim3((unsigned)blocks), dim3(256), 0, stream, n_seq, K, gamma,
                                     depth, tok, mult, ndist, key, ctx, pos, row_k, next_key, next_ctx, next_pos,
                                     next_k, child_node, node_key, node_ctx, node_pos);
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_hetero_expand(int32_t n_seq, int32_t B, int32_t gamma, int32_t depth, const int32_t* tok,
                                 const uint64_t* key, const uint64_t* ctx, const uint32_t* pos, const int32_t* owner,
                                 uint64_t* next_key, uint64_t* next_ctx, uint32_t* next_pos, int32_t* next_owner,
                                 int32_t* list_tok, int32_t* list_nd, int32_t* child_node, uint64_t* node_key,
                                 uint64_t* node_ctx, uint32_t* node_pos, cudaStream_t stream) {
    if (n_seq == 0) return cudaSuccess;
    const int64_t blocks = ((int64_t)n_seq * 32 + 255) / 256;
    const cudaError_t e = launch_pdl(hetero_expand_kernel, dim3((unsigned)blocks), dim3(256), 0, stream, n_seq, B,
                                     gamma, depth, tok, key, ctx, pos, owner, next_key, next_ctx, next_pos, next_owner,
                                     list_tok, list_nd, child_node, node_key, node_ctx, node_pos);
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_hetero_block(int64_t n, int32_t B, const int32_t* tok, const uint64_t* key, const uint64_t* ctx,
                                const uint32_t* pos, int32_t* out, cudaStream_t stream) {
    if (n == 0) return cudaSuccess;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 152 * 16) blocks = 152 * 16;
    hetero_block_kernel<<<(unsigned)blocks, 256, 0, stream>>>(n, B, tok, key, ctx, pos, out);
    return cudaGetLastError();
}

cudaError_t launch_words(const uint64_t* key, const uint64_t* ctx, const uint32_t* pos, int64_t n_rows, int64_t V,
                         int32_t arrival, uint32_t* out, cudaStream_t stream) {
    int64_t total = n_rows * V;
    if (total == 0) return cudaSuccess;
    int64_t blocks = (total + 255) / 256;
    if (blocks > 65535 * 8) blocks = 65535 * 8;
    words_kernel<<<(unsigned)blocks, 256, 0, stream>>>(key, ctx, pos, n_rows, V, arrival, out);
    return cudaGetLastError();
}

cudaError_t launch_selftest(uint64_t w_begin, uint64_t w_end, float* out, cudaStream_t stream) {
    if (w_end <= w_begin) return cudaSuccess;
    uint64_t n = w_end - w_begin;
    uint64_t blocks = (n + 255) / 256;
    if (blocks > 152 * 64) blocks = 152 * 64;
    selftest_kernel<<<(unsigned)blocks, 256, 0, stream>>>(w_begin, w_end, out);
    return cudaGetLastError();
}

cudaError_t launch_selftest_lg2(uint32_t b0, uint32_t b1, float* out, cudaStream_t stream) {
    if (b1 <= b0) return cudaSuccess;
    uint64_t blocks = ((uint64_t)(b1 - b0) + 255) / 256;
    if (blocks > 152 * 64) blocks = 152 * 64;
    selftest_lg2_kernel<<<(unsigned)blocks, 256, 0, stream>>>(b0, b1, out);
    return cudaGetLastError();
}

}  // namespace pps
