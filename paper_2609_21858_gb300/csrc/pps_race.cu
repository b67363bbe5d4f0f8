// pps_race.cu -- the fused keyed-race streaming kernel (draft lists and
// target winners) with the tree walk fused behind a per-sequence ticket.
//
// Work split.  The n_rows x vocab logits are viewed as one flattened range of
// 16-byte vectors (8 bf16 or 4 fp32 tokens); CTA b of G streams the slice
// [b*total/G, (b+1)*total/G), i.e. whole rows plus at most two partial rows.
// A row cut between CTAs is finished by the CTA that arrives last at the
// row's counter (no CTA ever waits on another).
//
// Per token (hot loop): the Philox word (row-specialised), the logit, and a
// conservative fp32 filter that rejects almost every token with one ex2 and
// an integer compare (pps_device.cuh).  Survivors get the accurate fp32 key
// and enter a per-warp sorted list of kp = min(32, 2k+2) entries (one entry
// per lane).  Lists are merged per CTA and per row with warp bitonic merges.
// The finished list proves its own completeness (every dropped token has a
// key above the k-th key plus both error bounds) and re-orders near-ties
// with the fp64 key s = ln E - l/T, so the selected tokens and their order
// are those of the exact definition (Alg. 2, Eq. 4, App. B algorithms).
#include <cfloat>
#include <climits>
#include <cstdint>

#include "pps.h"
#include "pps_device.cuh"
#include "pps_internal.h"

namespace pps {

#define FULL 0xffffffffu
constexpr float kInf = __builtin_huge_valf();

__device__ __forceinline__ bool lex_less(float ak, int ai, float bk, int bi) {
    return ak < bk || (ak == bk && ai < bi);
}
__device__ __forceinline__ bool lex_less_d(double ak, int ai, double bk, int bi) {
    return ak < bk || (ak == bk && ai < bi);
}

// ---------------------------------------------------------------- warp lists
// A warp list holds entries (k, i) sorted ascending by (k, i), entry m in
// lane m; lanes >= kp hold (+inf, INT_MAX).

// insert one warp-uniform entry (serial path for a few survivors)
__device__ __forceinline__ void list_insert(float& lk, int& li, float ck, int ci, int kp, int lane) {
    bool less = lane < kp && lex_less(ck, ci, lk, li);
    unsigned m = __ballot_sync(FULL, less);
    if (m == 0) return;
    int p = __ffs(m) - 1;
    float uk = __shfl_up_sync(FULL, lk, 1);
    int ui = __shfl_up_sync(FULL, li, 1);
    if (lane > p) {
        lk = uk;
        li = ui;
    } else if (lane == p) {
        lk = ck;
        li = ci;
    }
    if (lane >= kp) {
        lk = kInf;
        li = INT_MAX;
    }
}

// bitonic sort of one entry per lane, ascending
__device__ __forceinline__ void warp_sort(float& k, int& i, int lane) {
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            float ok = __shfl_xor_sync(FULL, k, stride);
            int oi = __shfl_xor_sync(FULL, i, stride);
            bool up = (lane & size) == 0 || size == 32;
            bool lower = (lane & stride) == 0;
            bool o_less = lex_less(ok, oi, k, i);
            bool take = (lower == up) ? o_less : (!o_less && !(ok == k && oi == i));
            if (take) {
                k = ok;
                i = oi;
            }
        }
    }
}

// merge a sorted list (lk, li) with a sorted batch (ok, oi); keep the kp smallest.
// Returns (warp-uniform) the smallest key it discards: the (kp+1)-th of the union.
template <bool TRACK>
__device__ __forceinline__ float warp_merge(float& lk, int& li, float ok, int oi, int kp, int lane) {
    float rk = __shfl_sync(FULL, ok, 31 - lane);
    int ri = __shfl_sync(FULL, oi, 31 - lane);
    float dropk = rk;
    if (lex_less(rk, ri, lk, li)) {
        dropk = lk;
        lk = rk;
        li = ri;
    }
    // (lk, li) is now bitonic and holds the 32 smallest of the union
#pragma unroll
    for (int stride = 16; stride > 0; stride >>= 1) {
        float xk = __shfl_xor_sync(FULL, lk, stride);
        int xi = __shfl_xor_sync(FULL, li, stride);
        bool lower = (lane & stride) == 0;
        bool o_less = lex_less(xk, xi, lk, li);
        if (lower ? o_less : (!o_less && !(xk == lk && xi == li))) {
            lk = xk;
            li = xi;
        }
    }
    if (TRACK) {
        if (kp < 32) dropk = fminf(dropk, __shfl_sync(FULL, lk, kp & 31));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) dropk = fminf(dropk, __shfl_xor_sync(FULL, dropk, o));
    }
    if (lane >= kp) {
        lk = kInf;
        li = INT_MAX;
    }
    return dropk;
}

__device__ __forceinline__ void warp_sort_d(double& k, int& i, int lane) {
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            double ok = __shfl_xor_sync(FULL, k, stride);
            int oi = __shfl_xor_sync(FULL, i, stride);
            bool up = (lane & size) == 0 || size == 32;
            bool lower = (lane & stride) == 0;
            bool o_less = lex_less_d(ok, oi, k, i);
            bool take = (lower == up) ? o_less : (!o_less && !(ok == k && oi == i));
            if (take) {
                k = ok;
                i = oi;
            }
        }
    }
}

// ---------------------------------------------------------------- logits

template <int DT>
__device__ __forceinline__ float load_logit(const void* row, int64_t i) {
    if (DT == 1) {
        unsigned short h = __ldg(reinterpret_cast<const unsigned short*>(row) + i);
        return __uint_as_float((uint32_t)h << 16);
    }
    return __ldg(reinterpret_cast<const float*>(row) + i);
}

__device__ __forceinline__ uint4 ldg_stream(const void* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

// ---------------------------------------------------------------- per-warp stream state

struct WarpList {
    float lk;   // this lane's entry
    int li;
    float th;   // key of entry kp-1 (+inf while not full)
    int thi;
    float tz;   // filter threshold (pps_device.cuh)
    int kp;

    __device__ __forceinline__ void reset(int kp_) {
        lk = kInf;
        li = INT_MAX;
        th = kInf;
        thi = INT_MAX;
        tz = kInf;
        kp = kp_;
    }
    __device__ __forceinline__ void refresh() {
        th = __shfl_sync(FULL, lk, kp - 1);
        thi = __shfl_sync(FULL, li, kp - 1);
        tz = filter_tz(th);
    }
};

// Offer the survivors of one vector (keys pk[e], token i0 + e) to the warp list.
template <int VW>
__device__ __forceinline__ void offer_survivors(WarpList& L, float (&pk)[VW], int64_t i0, int lane) {
    while (true) {
        float bk = kInf;
        int bi = INT_MAX, be = -1;
#pragma unroll
        for (int e = 0; e < VW; ++e) {
            if (lex_less(pk[e], (int)(i0 + e), bk, bi)) {
                bk = pk[e];
                bi = (int)(i0 + e);
                be = e;
            }
        }
        bool valid = be >= 0 && bk < kInf && lex_less(bk, bi, L.th, L.thi);
        unsigned vm = __ballot_sync(FULL, valid);
        if (vm == 0) break;
        if (__popc(vm) <= 3) {
            unsigned m = vm;
            while (m) {
                int src = __ffs(m) - 1;
                m &= m - 1;
                float ck = __shfl_sync(FULL, bk, src);
                int ci = __shfl_sync(FULL, bi, src);
                list_insert(L.lk, L.li, ck, ci, L.kp, lane);
            }
        } else {
            float ok = valid ? bk : kInf;
            int oi = valid ? bi : INT_MAX;
            warp_sort(ok, oi, lane);
            warp_merge<false>(L.lk, L.li, ok, oi, L.kp, lane);
        }
        if (valid) {
#pragma unroll
            for (int e = 0; e < VW; ++e)
                if (e == be) pk[e] = kInf;
        }
        L.refresh();
    }
}

// Process one 16-byte vector of tokens [i0, i0+VW) with words from RowPhilox.
template <int DT>
__device__ __forceinline__ void process_vector(WarpList& L, const RowPhilox& rp, uint4 d, int64_t vidx, int nvalid,
                                               float c, int lane) {
    constexpr int VW = DT == 1 ? 8 : 4;
    const int64_t i0 = vidx * VW;
    uint32_t w[VW];
    float l[VW];
    if constexpr (DT == 1) {
        uint4 b0 = rp.block((uint32_t)(2 * vidx));
        uint4 b1 = rp.block((uint32_t)(2 * vidx + 1));
        w[0] = b0.x; w[1] = b0.y; w[2] = b0.z; w[3] = b0.w;
        w[4] = b1.x; w[5] = b1.y; w[6] = b1.z; w[7] = b1.w;
        l[0] = bf16_lo(d.x); l[1] = bf16_hi(d.x); l[2] = bf16_lo(d.y); l[3] = bf16_hi(d.y);
        l[4] = bf16_lo(d.z); l[5] = bf16_hi(d.z); l[6] = bf16_lo(d.w); l[7] = bf16_hi(d.w);
    } else {
        uint4 b0 = rp.block((uint32_t)vidx);
        w[0] = b0.x; w[1] = b0.y; w[2] = b0.z; w[3] = b0.w;
        l[0] = __uint_as_float(d.x); l[1] = __uint_as_float(d.y);
        l[2] = __uint_as_float(d.z); l[3] = __uint_as_float(d.w);
    }
    unsigned m = 0;
#pragma unroll
    for (int e = 0; e < VW; ++e) m |= (unsigned)(filter_pass(w[e], l[e], c, L.tz) && e < nvalid) << e;
    if (__any_sync(FULL, m != 0)) {
        float pk[VW];
#pragma unroll
        for (int e = 0; e < VW; ++e) pk[e] = (m >> e & 1u) ? key32(w[e], l[e], c) : kInf;
        offer_survivors<VW>(L, pk, i0, lane);
    }
}

// ---------------------------------------------------------------- finalize

template <int DT>
__device__ __forceinline__ float logit_at(const RaceArgs& a, int64_t r, int64_t i) {
    const char* base = reinterpret_cast<const char*>(a.logits) + (size_t)r * (size_t)a.stride * (DT == 1 ? 2 : 4);
    return load_logit<DT>(base, i);
}

__device__ void walk_sequence(const RaceArgs& a, int s);

// Warp 0 finishes row r from its complete list (lk, li) and the drop bound.
template <int DT, bool VERIFY>
__device__ void finalize_row(const RaceArgs& a, int64_t r, float lk, int li, float theta_drop, int kr, int kp,
                             int lane) {
    const int nvalid = __popc(__ballot_sync(FULL, lane < kp && lk < kInf));
    const float tau = nvalid >= kr ? __shfl_sync(FULL, lk, kr - 1) : kInf;
    bool complete;
    if (nvalid < kr)
        complete = theta_drop == kInf;
    else if (tau == -kInf)
        complete = true;
    else
        complete = theta_drop == kInf || theta_drop > tau + key_err_bound(tau) + key_err_bound(theta_drop);
    if (lane == 0 && a.status) {
        unsigned f = complete ? 0u : PPS_FLAG_GUARD;
        if (nvalid >= kr && tau > -kInf && fabsf(tau) > 65536.0f) f |= PPS_FLAG_LOGIT_RANGE;
        if (f) atomicOr(a.status, f);
    }
    // near ties among the first min(nvalid, kr+1) entries
    float nk = __shfl_down_sync(FULL, lk, 1);
    int lim = min(nvalid, kr + 1);
    bool close = lane + 1 < lim && !(nk - lk > key_err_bound(lk) + key_err_bound(nk));
    const bool need_exact = (__ballot_sync(FULL, close) != 0) || (!VERIFY && a.iid);
    const uint64_t key = a.key[r], ctx = a.ctx[r];
    const uint32_t pos = a.pos[r];
    double dk = (double)INFINITY;
    float sk = key_to_s(lk);
    if (need_exact) {
        if (lane < nvalid) {
            uint32_t w = word_of(key, ctx, pos, li, 1);
            dk = key64(w, logit_at<DT>(a, r, li), a.T);
        }
        warp_sort_d(dk, li, lane);
        sk = (float)dk;
    }
    if (VERIFY) {
        int win = __shfl_sync(FULL, li, 0);
        if (nvalid == 0) win = -1;
        if (lane == 0) {
            a.out_winner[r] = win;
            a.out_word[r] = win >= 0 ? word_of(key, ctx, pos, win, 1) : 0u;
        }
        return;
    }
    const int K = a.K;
    const int nuse = min(nvalid, kr);
    const bool mine = lane < nuse;
    int tok = mine ? li : -1;
    int mult = mine ? 1 : 0;
    int sample = tok;
    if (a.iid) {
        // multi-arrival scores ln(G_{t,j}) - l_t/T of the nuse tokens, j = 1..kr;
        // the kr smallest (ties by token, then arrival) are the samples
        mult = 0;
        sample = -1;
        float lt = mine ? logit_at<DT>(a, r, li) : 0.0f;
        double G = mine ? exp1_f64(word_of(key, ctx, pos, li, 1)) : 0.0;
        double h = mine ? dk : (double)INFINITY;
        int j = 1;
        for (int m = 0; m < kr; ++m) {
            // warp argmin of (h, tok, j)
            double bh = h;
            int bt = mine ? tok : INT_MAX, bj = j, bl = lane;
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                double oh = __shfl_xor_sync(FULL, bh, off);
                int ot = __shfl_xor_sync(FULL, bt, off);
                int oj = __shfl_xor_sync(FULL, bj, off);
                int ol = __shfl_xor_sync(FULL, bl, off);
                bool better = oh < bh || (oh == bh && (ot < bt || (ot == bt && oj < bj)));
                if (better) {
                    bh = oh;
                    bt = ot;
                    bj = oj;
                    bl = ol;
                }
            }
            if (bt == INT_MAX) break;  // fewer usable tokens than samples
            if (lane == m) sample = bt;
            if (lane == bl) {
                ++mult;
                ++j;
                if (j <= kr) {
                    G += exp1_f64(word_of(key, ctx, pos, tok, j));
                    double ld = (double)lt;
                    h = log(G) - ld / (double)a.T;
                } else {
                    h = (double)INFINITY;
                }
            }
        }
    }
    const int nd = __popc(__ballot_sync(FULL, mult > 0));
    if (lane < K) {
        size_t o = (size_t)r * K + lane;
        a.out_tok[o] = lane < kr ? tok : -1;
        if (a.out_key) a.out_key[o] = (mine && lane < kr) ? sk : kInf;
        a.out_mult[o] = lane < kr ? mult : 0;
        if (a.out_samples) a.out_samples[o] = lane < kr ? sample : -1;
    }
    if (lane == 0) a.out_nd[r] = nd;
}

__device__ __forceinline__ int64_t cta_of(int64_t g, int64_t total, int G) {
    // largest b with floor(b*total/G) <= g
    return ((g + 1) * (int64_t)G - 1) / total;
}

__device__ __forceinline__ int seq_of_node(const int32_t* seq_off, int n_seq, int64_t r) {
    int lo = 0, hi = n_seq;  // find s with seq_off[s] <= r < seq_off[s+1]
    while (hi - lo > 1) {
        int mid = (lo + hi) >> 1;
        if (__ldg(seq_off + mid) <= r)
            lo = mid;
        else
            hi = mid;
    }
    return lo;
}

__device__ void walk_sequence(const RaceArgs& a, int s) {
    const int W = a.gamma + 1;
    int c = __ldg(a.seq_off + s);
    if (c < 0 || c >= a.n_rows) return;
    int acc = 0, ne = 0;
    double S = 0.0;
    bool stopped = false;
    for (int step = 0; step < a.gamma; ++step) {
        int y = __ldcg(a.out_winner + c);
        if (y < 0) {
            stopped = true;
            break;
        }
        double A = score64(__ldcg(a.out_word + c));
        a.out_em[(size_t)s * W + ne] = y;
        a.out_sc[(size_t)s * W + ne] = (float)A;
        S += A;
        ++ne;
        int dr = __ldg(a.node_draft_row + c), found = -1;
        if (dr >= 0 && dr < a.n_draft) {
            int nd = min(__ldg(a.draft_nd + dr), a.Kd);
            for (int m = 0; m < nd; ++m)
                if (__ldg(a.draft_tok + (size_t)dr * a.Kd + m) == y) {
                    found = m;
                    break;
                }
        }
        if (found < 0) {
            stopped = true;
            break;
        }
        int nxt = __ldg(a.child_node + (size_t)dr * a.Kd + found);
        if (nxt < 0 || nxt >= a.n_rows) {
            stopped = true;
            break;
        }
        c = nxt;
        ++acc;
    }
    if (!stopped) {
        int y = __ldcg(a.out_winner + c);
        if (y >= 0) {
            double A = score64(__ldcg(a.out_word + c));
            a.out_em[(size_t)s * W + ne] = y;
            a.out_sc[(size_t)s * W + ne] = (float)A;
            S += A;
            ++ne;
        }
    }
    for (int t = ne; t < W; ++t) {
        a.out_em[(size_t)s * W + t] = -1;
        a.out_sc[(size_t)s * W + t] = 0.0f;
    }
    a.out_acc[s] = acc;
    a.out_ne[s] = ne;
    a.out_ss[s] = S;
}

// ---------------------------------------------------------------- the kernel

template <int DT, bool VERIFY, bool VEC>
__global__ void __launch_bounds__(kThreads, 3) race_kernel(const RaceArgs a) {
    constexpr int VW = DT == 1 ? 8 : 4;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __shared__ float s_key[kWarps][32];
    __shared__ int s_idx[kWarps][32];
    __shared__ float s_theta[kWarps];

    const int64_t b = blockIdx.x;
    const int64_t g0 = b * a.total / a.G, g1 = (b + 1) * a.total / a.G;
    if (g0 >= g1) return;
    const float c = a.c;
    const int64_t nv = a.nv;
    const int tail = (int)(a.V - (nv - 1) * VW);  // tokens in the last vector of a row (1..VW)
    const size_t esz = DT == 1 ? 2 : 4;

    for (int64_t r = g0 / nv; r < a.n_rows && r * nv < g1; ++r) {
        const int64_t v0 = max(g0, r * nv) - r * nv, v1 = min(g1, (r + 1) * nv) - r * nv;
        int kr = 1;
        if (!VERIFY) {
            kr = a.row_k ? __ldg(a.row_k + r) : a.K;
            kr = max(1, min(kr, a.K));
        }
        const int kp = min(32, 2 * kr + 2);
        RowPhilox rp;
        rp.init(__ldg(a.key + r), __ldg(a.ctx + r), __ldg(a.pos + r));
        const char* row = reinterpret_cast<const char*>(a.logits) + (size_t)r * (size_t)a.stride * esz;

        WarpList L;
        L.reset(kp);
        // stream: thread t takes vectors v0 + t, v0 + t + kThreads, ...
        int64_t v = v0 + threadIdx.x;
        if (VEC) {
            const int64_t vfull_end = (tail == VW) ? v1 : min(v1, nv - 1);
            uint4 cur = make_uint4(0, 0, 0, 0), nxt = cur;
            if (v < vfull_end) cur = ldg_stream(row + (size_t)v * 16);
            // warps iterate in lockstep while any lane has work
            while (__any_sync(FULL, v < vfull_end)) {
                int64_t vn = v + kThreads;
                if (vn < vfull_end) nxt = ldg_stream(row + (size_t)vn * 16);
                int nvld = v < vfull_end ? VW : 0;
                process_vector<DT>(L, rp, cur, v < vfull_end ? v : 0, nvld, c, lane);
                cur = nxt;
                v = vn;
            }
            // ragged last vector of the row (scalar loads)
            if (vfull_end < v1) {
                int64_t vl = nv - 1;
                uint4 d = make_uint4(0, 0, 0, 0);
                int nvld = 0;
                if (threadIdx.x == (int)((vl - v0) % kThreads) && vl >= v0) {
                    uint32_t tmp[4] = {0u, 0u, 0u, 0u};
                    for (int e = 0; e < tail; ++e) {
                        int64_t i = vl * VW + e;
                        if (DT == 1) {
                            uint32_t h = __ldg(reinterpret_cast<const unsigned short*>(row) + i);
                            tmp[e >> 1] |= h << (16 * (e & 1));
                        } else {
                            tmp[e] = __float_as_uint(__ldg(reinterpret_cast<const float*>(row) + i));
                        }
                    }
                    d = make_uint4(tmp[0], tmp[1], tmp[2], tmp[3]);
                    nvld = tail;
                }
                process_vector<DT>(L, rp, d, nvld ? vl : 0, nvld, c, lane);
            }
        } else {
            // unaligned rows: scalar loads for every token
            while (__any_sync(FULL, v < v1)) {
                uint32_t tmp[4] = {0u, 0u, 0u, 0u};
                int nvld = 0;
                if (v < v1) {
                    nvld = (v == nv - 1) ? tail : VW;
                    for (int e = 0; e < nvld; ++e) {
                        int64_t i = v * VW + e;
                        if (DT == 1) {
                            uint32_t h = __ldg(reinterpret_cast<const unsigned short*>(row) + i);
                            tmp[e >> 1] |= h << (16 * (e & 1));
                        } else {
                            tmp[e] = __float_as_uint(__ldg(reinterpret_cast<const float*>(row) + i));
                        }
                    }
                }
                process_vector<DT>(L, rp, make_uint4(tmp[0], tmp[1], tmp[2], tmp[3]), nvld ? v : 0, nvld, c, lane);
                v += kThreads;
            }
        }

        // ---- merge the warp lists of this CTA
        s_key[warp][lane] = L.lk;
        s_idx[warp][lane] = L.li;
        if (lane == 0) s_theta[warp] = L.th;
        __syncthreads();
        if (warp == 0) {
            float lk = L.lk;
            int li = L.li;
            float theta_drop = s_theta[0];
            // every token left out of the merged list has a key >= theta_drop: the warps
            // dropped only keys >= their final kp-th key, the merges drop what they return
            for (int w = 1; w < kWarps; ++w) {
                float dk = warp_merge<true>(lk, li, s_key[w][lane], s_idx[w][lane], kp, lane);
                theta_drop = fminf(theta_drop, fminf(s_theta[w], dk));
            }
            bool final_here = v0 == 0 && v1 == nv;
            if (!final_here) {
                // publish this segment's list; the last CTA of the row merges all segments
                Partial* P = a.partials + (b + r);
                P->key[lane] = lk;
                P->idx[lane] = li;
                if (lane == 0) P->theta_drop = theta_drop;
                __threadfence();
                __syncwarp();
                const int64_t first_cta = cta_of(r * nv, a.total, a.G);
                const int64_t last_cta = cta_of(r * nv + nv - 1, a.total, a.G);
                unsigned last = 0;
                if (lane == 0) {
                    unsigned t = atomicAdd(a.row_cnt + r, 1u);
                    last = t == (unsigned)(last_cta - first_cta);
                    if (last) a.row_cnt[r] = 0u;
                }
                final_here = __shfl_sync(FULL, last, 0) != 0;
                if (final_here) {
                    __threadfence();
                    lk = kInf;
                    li = INT_MAX;
                    theta_drop = kInf;
                    for (int64_t bb = first_cta; bb <= last_cta; ++bb) {
                        const Partial* Q = a.partials + (bb + r);
                        float dk = warp_merge<true>(lk, li, __ldcg(Q->key + lane), __ldcg(Q->idx + lane), kp, lane);
                        theta_drop = fminf(theta_drop, fminf(__ldcg(&Q->theta_drop), dk));
                    }
                }
            }
            if (final_here) {
                finalize_row<DT, VERIFY>(a, r, lk, li, theta_drop, kr, kp, lane);
                if constexpr (VERIFY) {
                    // sequence ticket: the CTA that finishes a sequence's last node walks it
                    __threadfence();
                    if (lane == 0) {
                        int s = seq_of_node(a.seq_off, a.n_seq, r);
                        int nn = __ldg(a.seq_off + s + 1) - __ldg(a.seq_off + s);
                        unsigned t = atomicAdd(a.seq_cnt + s, 1u);
                        if (t == (unsigned)(nn - 1)) {
                            a.seq_cnt[s] = 0u;
                            __threadfence();
                            walk_sequence(a, s);
                        }
                    }
                }
            }
        }
        __syncthreads();
    }
}

int race_grid(int64_t total, int dtype, bool verify, bool vec) {
    static int sms = 0, occ[2][2][2] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (sms == 0) {
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (sms <= 0) sms = 1;
    }
    int& o = occ[dtype][verify][vec];
    if (o == 0) {
        const void* fn = nullptr;
        if (dtype == 1)
            fn = verify ? (vec ? (const void*)race_kernel<1, true, true> : (const void*)race_kernel<1, true, false>)
                        : (vec ? (const void*)race_kernel<1, false, true> : (const void*)race_kernel<1, false, false>);
        else
            fn = verify ? (vec ? (const void*)race_kernel<0, true, true> : (const void*)race_kernel<0, true, false>)
                        : (vec ? (const void*)race_kernel<0, false, true> : (const void*)race_kernel<0, false, false>);
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, fn, kThreads, 0);
        if (o <= 0) o = 1;
    }
    int64_t g = (int64_t)sms * o;
    int64_t by_size = (total + kMinVecsPerCta - 1) / kMinVecsPerCta;
    if (by_size < g) g = by_size;
    if (g > kGridMax) g = kGridMax;
    if (g < 1) g = 1;
    return (int)g;
}

cudaError_t launch_race(const RaceArgs& a, int dtype, bool verify, bool vec, cudaStream_t stream) {
    dim3 grid(a.G), block(kThreads);
    if (dtype == 1) {
        if (verify) {
            if (vec) race_kernel<1, true, true><<<grid, block, 0, stream>>>(a);
            else race_kernel<1, true, false><<<grid, block, 0, stream>>>(a);
        } else {
            if (vec) race_kernel<1, false, true><<<grid, block, 0, stream>>>(a);
            else race_kernel<1, false, false><<<grid, block, 0, stream>>>(a);
        }
    } else {
        if (verify) {
            if (vec) race_kernel<0, true, true><<<grid, block, 0, stream>>>(a);
            else race_kernel<0, true, false><<<grid, block, 0, stream>>>(a);
        } else {
            if (vec) race_kernel<0, false, true><<<grid, block, 0, stream>>>(a);
            else race_kernel<0, false, false><<<grid, block, 0, stream>>>(a);
        }
    }
    return cudaGetLastError();
}

}  // namespace pps
