// pps_race.cu -- the fused keyed-race streaming kernel (draft lists and
// target winners) with the tree walk fused behind a per-sequence ticket.
//
// Work split.  The n_rows x vocab logits are viewed as one flattened range of
// 16-byte vectors (8 bf16 or 4 fp32 tokens).  A CTA is a single warp; warp gw
// of NW streams the slice [gw*total/NW, (gw+1)*total/NW), i.e. a few whole
// rows plus at most two partial rows.  A row cut between warps is merged and
// finished by the warp that arrives last at the row's counter; a sequence's
// walk is run by the warp that finishes its last node.  No warp ever waits
// for another and the kernel has no block-wide barrier.  One-warp CTAs also
// make every per-row value warp-uniform, so the Philox round keys of a row
// can live in uniform registers.
//
// Per token (fast loop): the Philox word (row-specialised), the logit, and a
// conservative fp32 filter that rejects almost every token with one ex2 and
// a few multiply-pipe operations (pps_device.cuh).  Survivors get the fp32 key
// and enter a per-warp sorted list of kp = min(32, 2k+1) entries (one per
// lane).  Lists of a row are merged with warp bitonic merges.  The finished
// list proves its own completeness (every dropped token has a key above the
// k-th key plus both error bounds) and re-orders near-ties with the fp64 key
// s = ln E - l/T, so the selected tokens and their order are those of the
// exact definition (Alg. 2, Eq. 4, App. B algorithms).
#include <cuda.h>

#include <atomic>
#include <cfloat>
#include <cstring>
#include <climits>
#include <cstdint>

#include "pps.h"
#include "pps_device.cuh"
#include "pps_internal.h"

#ifndef PPS_UNITS
#define PPS_UNITS 3  // 8-token units per lane per fast-loop iteration (2 Philox blocks each), draft rows
#endif
#ifndef PPS_UNITS_VERIFY
#define PPS_UNITS_VERIFY 3  // the same for verify rows and one-token draft rows
#endif
#ifndef PPS_PREFETCH
#define PPS_PREFETCH 0  // 1: load the next iteration's vectors one iteration ahead (costs registers)
#endif
#ifndef PPS_ROWBOUND
#define PPS_ROWBOUND 1  // 1: warps that share a row share its filter bound through the workspace
#endif
#ifndef PPS_IID_FAST
#define PPS_IID_FAST 1  // 1: IID epilogue in fp32 with a separation check (fp64 only on near ties)
#endif
#ifndef PPS_VECFILTER
#define PPS_VECFILTER 1  // 1: one filter test per 16-byte vector on verify rows and fp32 rows
#endif
#ifndef PPS_PACKED
#define PPS_PACKED 0  // 1: pairs of filter sums with packed fp32x2 fma/add
#endif
#ifndef PPS_RACE_MIN_BLOCKS
#define PPS_RACE_MIN_BLOCKS 16  // one-warp CTAs resident per SM (register budget 128, no spills)
#endif
#ifndef PPS_BLOCK_MIN_BLOCKS
#define PPS_BLOCK_MIN_BLOCKS 12  // the same for proposal rows of the augmented race (16 spills)
#endif
#ifndef PPS_VF_MAXK
#define PPS_VF_MAXK 4  // draft rows with lists up to this long stream like verify rows (one test per vector)
#endif
#ifndef PPS_SEG_CAP
#define PPS_SEG_CAP 30  // at most this many warp segments per row (small launches; keeps <= 32 partial lists)
#endif

namespace pps {

#define FULL 0xffffffffu
constexpr float kInf = __builtin_huge_valf();

// Shared row bound: a float kept as ~(order-preserving bits), so that atomicMax
// keeps the smallest bound and the zeroed word reads as none (+inf).
__device__ __forceinline__ uint32_t bound_enc(float f) {
    const uint32_t b = __float_as_uint(f);
    return ~((b & 0x80000000u) ? ~b : (b | 0x80000000u));
}
__device__ __forceinline__ float bound_dec(uint32_t e) {
    if (e == 0u) return kInf;
    const uint32_t o = ~e;
    return __uint_as_float((o & 0x80000000u) ? (o & 0x7fffffffu) : ~o);
}

__device__ __forceinline__ bool lex_less(float ak, int ai, float bk, int bi) {
    return ak < bk || (ak == bk && ai < bi);
}
__device__ __forceinline__ bool lex_less_d(double ak, int ai, double bk, int bi) {
    return ak < bk || (ak == bk && ai < bi);
}

// fp32 key -> unsigned integer with the same order (-0 taken as +0), and back,
// so that a warp argmin of (key, token) is two redux.min instructions.
__device__ __forceinline__ uint32_t ord_key(float f) {
    const uint32_t b = __float_as_uint(f + 0.0f);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float unord_key(uint32_t u) {
    return __uint_as_float((u & 0x80000000u) ? (u & 0x7fffffffu) : ~u);
}
// Warp argmin of (key, token) by lexicographic order; tokens are non-negative
// (INT_MAX: empty).  Returns the winning token (INT_MAX when every lane is
// empty) and its key in bk.
__device__ __forceinline__ int warp_argmin(float k, int t, float& bk) {
    const uint32_t u = ord_key(k);
    const uint32_t mu = __reduce_min_sync(FULL, u);
    const uint32_t mt = __reduce_min_sync(FULL, u == mu ? (uint32_t)t : 0xffffffffu);
    bk = unord_key(mu);
    return (int)mt;
}

// ---------------------------------------------------------------- warp lists
// A warp list holds entries (k, i) sorted ascending by (k, i), entry m in
// lane m; lanes >= kp hold (+inf, INT_MAX).

// insert one warp-uniform entry (serial path for a few survivors); returns
// the key left out: the entry pushed out of a full list (+inf if there was
// room), or ck itself when it does not enter
__device__ __forceinline__ float list_insert(float& lk, int& li, float ck, int ci, int kp, int lane) {
    bool less = lane < kp && lex_less(ck, ci, lk, li);
    unsigned m = __ballot_sync(FULL, less);
    if (m == 0) return ck;
    const float last = __shfl_sync(FULL, lk, kp - 1);
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
    return last;
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

// scalar load of the tokens of vector v (i < V), packed like a 16-byte vector
template <int DT>
__device__ __forceinline__ uint4 load_scalar(const char* row, int64_t v, int64_t V) {
    constexpr int VW = DT == 1 ? 8 : 4;
    uint32_t t[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int e = 0; e < VW; ++e) {
        int64_t i = v * VW + e;
        if (i < V) {
            if constexpr (DT == 1) {
                uint32_t h = __ldg(reinterpret_cast<const unsigned short*>(row) + i);
                t[e >> 1] |= h << (16 * (e & 1));
            } else {
                t[e] = __float_as_uint(__ldg(reinterpret_cast<const float*>(row) + i));
            }
        }
    }
    return make_uint4(t[0], t[1], t[2], t[3]);
}

// Counter offset of block b of a lane's fast-loop iteration: bf16 blocks come
// in pairs (2v, 2v+1) of one vector v, vectors 32 apart; fp32 blocks are
// single vectors 32 apart.
template <int DT>
__device__ __forceinline__ uint32_t block_offset(int b) {
    return DT == 1 ? (uint32_t)((b >> 1) * 64 + (b & 1)) : (uint32_t)(32 * b);
}

// the four logits of block b of an iteration's vectors d[]
template <int DT, int N>
__device__ __forceinline__ void block_logits(const uint4 (&d)[N], int b, float (&l)[4]) {
    if constexpr (DT == 1) {
        const uint4 v = d[b >> 1];
        const uint32_t x0 = (b & 1) ? v.z : v.x, x1 = (b & 1) ? v.w : v.y;
        l[0] = bf16_lo(x0);
        l[1] = bf16_hi(x0);
        l[2] = bf16_lo(x1);
        l[3] = bf16_hi(x1);
    } else {
        const uint4 v = d[b];
        l[0] = __uint_as_float(v.x);
        l[1] = __uint_as_float(v.y);
        l[2] = __uint_as_float(v.z);
        l[3] = __uint_as_float(v.w);
    }
}

// ---------------------------------------------------------------- per-warp list state

struct WarpList {
    float lk;  // this lane's entry
    int li;
    float th;  // key of entry kp-1 (+inf while not full)
    int thi;
    float tf;  // filter bound: the filter drops only tokens with keys >= tf; never rises
    float tz;  // filter threshold for tf (pps_device.cuh)
    float mr;  // smallest key of a survivor the list left out (rejected or pushed out)
    int kp;
    int k;     // entries the row needs (kp > k leaves room for near ties)

    __device__ __forceinline__ void reset(int kp_, int k_) {
        lk = kInf;
        li = INT_MAX;
        th = kInf;
        thi = INT_MAX;
        tf = kInf;
        tz = kInf;
        mr = kInf;
        kp = kp_;
        k = k_;
    }
    // lower tf to b (no effect when b >= tf); the filter tests plain keys
    // against tf + shift (shift = 0 except for proposal rows of the augmented race)
    __device__ __forceinline__ void bound(float b, float shift = 0.f) {
        tf = fminf(tf, b);
        tz = filter_tz(tf + shift);
    }
    // after the list changed: tf <= min(th, (entry k-1) + filter_slack), the
    // slack widened by 4 eb for keys with extra error eb.  A list with no
    // spare entry (kp = k, i.e. k = 32) keeps tf at the slack bound instead:
    // the filter passes the keys between entry kp-1 and it, the list leaves
    // them out and records the smallest in mr, so such a list still proves
    // itself complete unless entry k and the next key nearly tie.
    __device__ __forceinline__ bool tight() const { return kp == k; }
    __device__ __forceinline__ void refresh(float shift = 0.f, float eb = 0.f) {
        th = __shfl_sync(FULL, lk, kp - 1);
        thi = __shfl_sync(FULL, li, kp - 1);
        const float sl = filter_slack(__shfl_sync(FULL, lk, k - 1)) + 4.0f * eb;
        bound(tight() ? sl : fminf(th, sl), shift);
    }
    // every token of the segment left out of the list has a key >= drop()
    __device__ __forceinline__ float drop() const { return fminf(tight() ? mr : th, tf); }
};

// Publish filter_slack of the list's k-th key (widened by eb) as a filter bound
// for every warp of the row: the row's k-th key is at most this list's, so
// the bound passes the completeness test of any segment that adopts it.
__device__ __forceinline__ void publish_bound(uint32_t* slot, const WarpList& L, float eb, int lane) {
    const float pub = filter_slack(__shfl_sync(FULL, L.lk, L.k - 1)) + eb * 4.0f;
    if (lane == 0 && pub < kInf) atomicMax(slot, bound_enc(pub));
}

// Offer the keyed survivors of one lane (pk[e] for token i0 + e, +inf = none)
// to the warp list: each round every lane offers its smallest remaining key
// below the threshold; up to three offers are inserted one by one, more are
// sorted across the warp and merged.  Ends when no lane has a key below it,
// so the threshold is always current.
template <int VW>
__device__ __forceinline__ void offer_survivors(WarpList& L, float (&pk)[VW], int64_t i0, int lane,
                                                float shift = 0.f, float eb = 0.f) {
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
        const bool valid = be >= 0 && bk < kInf && lex_less(bk, bi, L.th, L.thi);
        const unsigned vm = __ballot_sync(FULL, valid);
        if (vm == 0) break;
        if (__popc(vm) <= 3) {
            unsigned m = vm;
            while (m) {
                const int src = __ffs(m) - 1;
                m &= m - 1;
                const float ck = __shfl_sync(FULL, bk, src);
                const int ci = __shfl_sync(FULL, bi, src);
                L.mr = fminf(L.mr, list_insert(L.lk, L.li, ck, ci, L.kp, lane));
            }
        } else {
            float ok = valid ? bk : kInf;
            int oi = valid ? bi : INT_MAX;
            warp_sort(ok, oi, lane);
            if (L.tight())
                L.mr = fminf(L.mr, warp_merge<true>(L.lk, L.li, ok, oi, L.kp, lane));
            else
                warp_merge<false>(L.lk, L.li, ok, oi, L.kp, lane);
        }
        // every offer of this round is now in the list or recorded in mr
#pragma unroll
        for (int e = 0; e < VW; ++e)
            if (e == be) pk[e] = kInf;
        L.refresh(shift, eb);
    }
    // keys not offered (at or above entry kp-1) are left out too
    float rem = kInf;
#pragma unroll
    for (int e = 0; e < VW; ++e) rem = fminf(rem, pk[e]);
    if (L.tight() && __any_sync(FULL, rem < kInf)) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) rem = fminf(rem, __shfl_xor_sync(FULL, rem, o));
        L.mr = fminf(L.mr, rem);
    }
}

// Filter, key and offer the 4 tokens of one Philox block (counter cb, tokens
// 4cb..4cb+3, logits l[]) for the lanes with `mine`.  BLK: the rows are
// proposal b's race over block b of the augmented source; survivors of the
// (shifted) plain filter are keyed with their block arrival (fp32, error
// bound widened by kBlkErr).
template <bool BLK>
__device__ __forceinline__ void block_survivors(WarpList& L, const RowPhilox& rp, bool mine, uint32_t cb,
                                                const float (&l)[4], unsigned valid, float c, int lane, const Blk& bk,
                                                uint64_t key, uint64_t ctx, uint32_t pos, uint32_t* slot) {
    float pk[4] = {kInf, kInf, kInf, kInf};
    if (mine) {
        const uint4 q = rp.block(cb);
        const uint32_t wq[4] = {q.x, q.y, q.z, q.w};
        unsigned pm = 0;
#pragma unroll
        for (int e = 0; e < 4; ++e)
            if (((valid >> e) & 1u) && filter_pass(wq[e], l[e], c, L.tz)) pm |= 1u << e;
        if constexpr (BLK) {
            if (pm) {
                // the block's J words and block-b excess words, four tokens per Philox block
                const uint64_t kj = key ^ kBlockJ, kf = key ^ ((uint64_t)(uint32_t)(bk.b + 1) * kBlockF);
                const uint4 jq = philox(cb, pos, (uint32_t)ctx, (uint32_t)(ctx >> 32), (uint32_t)kj,
                                        (uint32_t)(kj >> 32));
                const uint4 fq = philox(cb, pos, (uint32_t)ctx, (uint32_t)(ctx >> 32), (uint32_t)kf,
                                        (uint32_t)(kf >> 32));
                const uint32_t wj[4] = {jq.x, jq.y, jq.z, jq.w}, wf[4] = {fq.x, fq.y, fq.z, fq.w};
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if ((pm >> e) & 1u)
                        pk[e] = block_key32(wq[e], block_j(wj[e], bk.B), wf[e], bk.b, bk.invB(), l[e], c);
            }
        } else {
#pragma unroll
            for (int e = 0; e < 4; ++e)
                if ((pm >> e) & 1u) pk[e] = key32(wq[e], l[e], c);
        }
    }
    offer_survivors<4>(L, pk, (int64_t)4 * cb, lane, BLK ? bk.shift() : 0.f, BLK ? kBlkErr : 0.f);
    if (slot != nullptr) publish_bound(slot, L, BLK ? kBlkErr : 0.f, lane);
}

// ---------------------------------------------------------------- rare paths (out of line)

struct SlowState {
    WarpList L;
};

// Blocks flagged by the fast scan wait in a per-warp queue of Philox block
// counters in shared memory (one iteration adds at most 32 x 2 x units).
constexpr int kMaxUnits = PPS_UNITS > PPS_UNITS_VERIFY ? PPS_UNITS : PPS_UNITS_VERIFY;
constexpr int kQueueCap = 32 + 32 * 2 * kMaxUnits;
static_assert(kQueueCap >= 1 + 2 * 96, "the queue also serves as the scratch of rescan_row");

// Work off the queue: lane j regenerates the words of queued block j (32 at
// a time), reloads its four logits, keys the tokens over the filter cut and
// offers them.  Out of line; the fast scan itself makes no calls.
template <int DT, bool BLK>
__device__ __noinline__ SlowState flush_queue(SlowState st, const uint32_t* q, int qn, const char* row, float c,
                                              uint64_t key, uint64_t ctx, uint32_t pos, Blk bk, uint32_t* slot) {
    const int lane = threadIdx.x & 31;
    RowPhilox rp;
    rp.init(key, ctx, pos);
    __syncwarp();
    for (int base = 0; base < qn; base += 32) {
        const bool mine = base + lane < qn;
        const uint32_t cb = mine ? q[base + lane] : 0u;
        float l[4] = {0.f, 0.f, 0.f, 0.f};
        if (mine) {
            if constexpr (DT == 1) {
                const uint2 v = __ldg(reinterpret_cast<const uint2*>(row) + cb);
                l[0] = bf16_lo(v.x);
                l[1] = bf16_hi(v.x);
                l[2] = bf16_lo(v.y);
                l[3] = bf16_hi(v.y);
            } else {
                const uint4 v = __ldg(reinterpret_cast<const uint4*>(row) + cb);
                l[0] = __uint_as_float(v.x);
                l[1] = __uint_as_float(v.y);
                l[2] = __uint_as_float(v.z);
                l[3] = __uint_as_float(v.w);
            }
        }
        block_survivors<BLK>(st.L, rp, mine, cb, l, 0xfu, c, lane, bk, key, ctx, pos, slot);
    }
    __syncwarp();
    return st;
}

// Scalar-load path, one vector per lane at a time: the last partial
// iteration of a segment, the ragged vector of a row, and unaligned rows.
// Tokens with a logit below `floor` take no part (-inf: none excluded).
template <int DT, bool BLK = false>
__device__ __noinline__ SlowState tail_loop(SlowState st, const char* row, int64_t V, int64_t base, int64_t v1,
                                            float c, uint64_t key, uint64_t ctx, uint32_t pos, float floor,
                                            Blk bk = Blk{}, uint32_t* slot = nullptr) {
    constexpr int VW = DT == 1 ? 8 : 4;
    const int lane = threadIdx.x & 31;
    RowPhilox rp;
    rp.init(key, ctx, pos);
    for (; base < v1; base += 32) {
        const int64_t v = base + lane;
        uint4 dv = make_uint4(0, 0, 0, 0);
        unsigned valid = 0;
        if (v < v1) {
            dv = load_scalar<DT>(row, v, V);
            const int64_t nt = min((int64_t)VW, V - v * VW);
            valid = (1u << nt) - 1u;
        }
        const uint4 d[2] = {dv, dv};
        // the vector's blocks: bf16 2 (counters 2v, 2v+1), fp32 1 (counter v)
#pragma unroll
        for (int h = 0; h < (DT == 1 ? 2 : 1); ++h) {
            unsigned vh = (valid >> (4 * h)) & 0xfu;
            float l[4];
            block_logits<DT>(d, h, l);
#pragma unroll
            for (int e = 0; e < 4; ++e)
                if (l[e] < floor) vh &= ~(1u << e);
            const uint32_t cb = DT == 1 ? (uint32_t)(2 * v + h) : (uint32_t)v;
            // any token of the block over the cut?
            bool pass = false;
            if (vh) {
                const uint4 q = rp.block(cb);
                const uint32_t wq[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) pass |= ((vh >> e) & 1u) && filter_pass(wq[e], l[e], c, st.L.tz);
            }
            if (__any_sync(FULL, pass))
                block_survivors<BLK>(st.L, rp, pass, cb, l, vh, c, lane, bk, key, ctx, pos, slot);
        }
    }
    return st;
}

// A filter bound for an empty list.  Lane j keys exactly (key32, the list's
// own key) the 8 tokens of its first unit of the segment's first fast
// iteration and keeps its smallest; the bound is filter_slack of the k-th
// smallest of the 32 lane minima.  Those k tokens lie in the segment, so the
// row's k-th key is at most their largest, and the slack keeps every token
// that could tie with it (tf itself is recorded as a drop bound).  Without
// it every block of the first iteration would pass the filter and be queued.
// BLK: the lane's smallest plain key is replaced by that token's block key.
template <int DT, bool BLK>
__device__ __noinline__ float seed_theta(const char* row, int64_t v0, float c, uint64_t key, uint64_t ctx,
                                         uint32_t pos, int k, Blk blk) {
    const int lane = threadIdx.x & 31;
    RowPhilox rp;
    rp.init(key, ctx, pos);
    const uint4* p = reinterpret_cast<const uint4*>(row) + v0 + lane;
    uint4 d[2];
    d[0] = __ldg(p);
    d[1] = DT == 1 ? d[0] : __ldg(p + 32);
    const uint32_t cl = DT == 1 ? (uint32_t)(2 * (v0 + lane)) : (uint32_t)(v0 + lane);
    float bk = kInf;
    int bi = INT_MAX;
#pragma unroll
    for (int b = 0; b < 2; ++b) {
        const uint32_t cb = cl + block_offset<DT>(b);
        const uint4 q = rp.block(cb);
        const uint32_t wq[4] = {q.x, q.y, q.z, q.w};
        float l[4];
        block_logits<DT>(d, b, l);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float k = key32(wq[e], l[e], c);
            const int i = (int)(4 * cb + e);
            if (lex_less(k, i, bk, bi)) {
                bk = k;
                bi = i;
            }
        }
    }
    if constexpr (BLK)
        bk = block_key_of(key, ctx, pos, bi, word_of(key, ctx, pos, bi, 1), load_logit<DT>(row, bi), c, blk.b,
                          blk.B, blk.invB());
    warp_sort(bk, bi, lane);
    return filter_slack(__shfl_sync(FULL, bk, k - 1)) + (BLK ? 4.0f * kBlkErr : 0.f);
}

// ---------------------------------------------------------------- the fast loop

// filter sums of the four tokens of one block, max of the four
__device__ __forceinline__ float block_filter_max(const uint4& w, const float (&l)[4], float c, float tz) {
#if PPS_PACKED
    float z0, z1, z2, z3;
    asm("{\n\t.reg .b64 a, b, t, d;\n\t"
        "mov.b64 a, {%4, %5};\n\tmov.b64 b, {%8, %8};\n\tmov.b64 t, {%9, %9};\n\t"
        "fma.rn.f32x2 d, a, b, t;\n\tmov.b64 {%0, %1}, d;\n\t"
        "mov.b64 a, {%6, %7};\n\tfma.rn.f32x2 d, a, b, t;\n\tmov.b64 {%2, %3}, d;\n\t}"
        : "=f"(z0), "=f"(z1), "=f"(z2), "=f"(z3)
        : "f"(l[0]), "f"(l[1]), "f"(l[2]), "f"(l[3]), "f"(c), "f"(tz));
    const float t0 = ex2_approx(z0), t1 = ex2_approx(z1), t2 = ex2_approx(z2), t3 = ex2_approx(z3);
    float s0, s1, s2, s3;
    asm("{\n\t.reg .b64 a, b, d;\n\t"
        "mov.b64 a, {%4, %5};\n\tmov.b64 b, {%8, %9};\n\tadd.rn.f32x2 d, a, b;\n\tmov.b64 {%0, %1}, d;\n\t"
        "mov.b64 a, {%6, %7};\n\tmov.b64 b, {%10, %11};\n\tadd.rn.f32x2 d, a, b;\n\tmov.b64 {%2, %3}, d;\n\t}"
        : "=f"(s0), "=f"(s1), "=f"(s2), "=f"(s3)
        : "f"(t0), "f"(t1), "f"(t2), "f"(t3), "f"(filter_word(w.x)), "f"(filter_word(w.y)),
          "f"(filter_word(w.z)), "f"(filter_word(w.w)));
    return fmaxf(fmaxf(s0, s1), fmaxf(s2, s3));
#else
    const float m01 = fmaxf(filter_sum(w.x, l[0], c, tz), filter_sum(w.y, l[1], c, tz));
    const float m23 = fmaxf(filter_sum(w.z, l[2], c, tz), filter_sum(w.w, l[3], c, tz));
    return fmaxf(m01, m23);
#endif
}

// Fast scan over iterations [it0, n_it) of the full vectors starting at
// vector v0 of a row.  Each iteration covers U x 32 (bf16) or x 64 (fp32)
// vectors; every lane takes U units of 8 tokens = 2 x U Philox blocks with
// counters cl + block_offset(b), cl advancing by 64 x U, so that many
// independent multiply chains are in flight per
// lane.  A lane keeps only the per-block maxima of the filter sums; a block
// with a token over the cut is appended to the warp's queue.  The scan makes
// no calls: it returns the iteration after which the queue holds 32 or more
// blocks (n_it when it ran to the end), so that nothing it keeps in
// registers (the row's round keys above all) lives across a call.
// VF: test each 16-byte vector once (verify rows, where one key is kept, and
// fp32 rows); otherwise each Philox block's four tokens (the vector test
// passes up to 8x more often under the looser bound of a K-list).
// slot (nullable): the row's shared bound, read every iteration; a smaller one
// lowers the filter threshold and is returned in tfa (the caller records it as
// this segment's drop bound).
template <int DT, bool VF, int U>
__device__ __forceinline__ int64_t fast_scan(const RowPhilox& rp, const char* row, int64_t v0, int64_t it0,
                                             int64_t n_it, float c, float tz, uint32_t* q, int& qn,
                                             const uint32_t* slot, float shift, float& tfa) {
    constexpr int NB = 2 * U;                  // Philox blocks per lane per iteration
    constexpr int ND = DT == 1 ? NB / 2 : NB;  // 16-byte vectors per lane per iteration
    constexpr int STEP = 32 * ND;              // vectors per iteration
    const int lane = threadIdx.x & 31;
    const uint4* p = reinterpret_cast<const uint4*>(row) + v0 + it0 * STEP + lane;
    uint32_t cl = (DT == 1 ? (uint32_t)(2 * (v0 + lane)) : (uint32_t)(v0 + lane)) + (uint32_t)(it0 * 64 * U);
#if PPS_PREFETCH
    uint4 nx[ND];
#pragma unroll
    for (int k = 0; k < ND; ++k) nx[k] = ldg_stream(p + 32 * k);
#endif
    for (int64_t it = it0; it < n_it; ++it) {
        uint4 d[ND];
#if PPS_PREFETCH
#pragma unroll
        for (int k = 0; k < ND; ++k) d[k] = nx[k];
        p += STEP;
        if (it + 1 < n_it) {
#pragma unroll
            for (int k = 0; k < ND; ++k) nx[k] = ldg_stream(p + 32 * k);
        }
#else
#pragma unroll
        for (int k = 0; k < ND; ++k) d[k] = ldg_stream(p + 32 * k);
        p += STEP;
#endif
        uint32_t shared_bound = 0u;
        if (slot != nullptr) asm volatile("ld.global.cg.u32 %0, [%1];" : "=r"(shared_bound) : "l"(slot));
        unsigned bm = 0;
        if constexpr (VF && PPS_VECFILTER) {
            // One test per 16-byte vector: the filter sum rises with the word and
            // the logit, so the vector's largest word with its largest logit
            // passes whenever one of its tokens would; the ex2 error is taken at
            // the larger argument, as in the per-token test, so the same margin
            // covers it.  A passing vector queues its Philox blocks for the
            // per-token test.
#pragma unroll
            for (int k = 0; k < ND; ++k) {
                if constexpr (DT == 1) {
                    const uint4 w0 = rp.block(cl + block_offset<DT>(2 * k));
                    const uint4 w1 = rp.block(cl + block_offset<DT>(2 * k + 1));
                    const uint32_t wm =
                        max(max(max(w0.x, w0.y), max(w0.z, w0.w)), max(max(w1.x, w1.y), max(w1.z, w1.w)));
                    const uint32_t m2 = bf2_max(bf2_max(d[k].x, d[k].y), bf2_max(d[k].z, d[k].w));
                    const float lm = fmaxf(bf16_lo(m2), bf16_hi(m2));
                    bm |= (filter_pass(wm, lm, c, tz) ? 3u : 0u) << (2 * k);
                } else {
                    const uint4 w = rp.block(cl + block_offset<DT>(k));
                    const uint32_t wm = max(max(w.x, w.y), max(w.z, w.w));
                    const float lm = fmaxf(fmaxf(__uint_as_float(d[k].x), __uint_as_float(d[k].y)),
                                           fmaxf(__uint_as_float(d[k].z), __uint_as_float(d[k].w)));
                    bm |= (filter_pass(wm, lm, c, tz) ? 1u : 0u) << k;
                }
            }
        } else {
#pragma unroll
            for (int b = 0; b < NB; ++b) {
                const uint4 w = rp.block(cl + block_offset<DT>(b));
                float l[4];
                block_logits<DT>(d, b, l);
                bm |= (unsigned)(block_filter_max(w, l, c, tz) >= kFilterCut) << b;
            }
        }
        if (slot != nullptr) {
            const float g = bound_dec(shared_bound);
            if (g < tfa) {
                tfa = g;
                tz = filter_tz(g + shift);
            }
        }
        if (__any_sync(FULL, bm != 0)) {
            // append this lane's flagged blocks at its offset in the warp's batch
            const int n = __popc(bm);
            int off = n;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int t = __shfl_up_sync(FULL, off, o);
                if (lane >= o) off += t;
            }
            const int total = __shfl_sync(FULL, off, 31);
            off += qn - n;
#pragma unroll
            for (int b = 0; b < NB; ++b)
                if ((bm >> b) & 1u) q[off++] = cl + block_offset<DT>(b);
            qn += total;
            if (qn >= 32) return it + 1;
        }
        cl += 64 * U;
    }
    return n_it;
}

// Stream vectors [v0, v1) of one row through the warp's list: full
// iterations through the fast loop, the rest through the scalar tail.
template <int DT, bool VEC, bool BLK, bool VF, int U>
__device__ __forceinline__ void stream_segment(WarpList& L, const char* row, int64_t V, int64_t v0, int64_t v1,
                                               float c, uint64_t key, uint64_t ctx, uint32_t pos, uint32_t* q,
                                               const Blk& bk, uint32_t* slot) {
    constexpr int VW = DT == 1 ? 8 : 4;
    constexpr int STEP = (DT == 1 ? 32 : 64) * U;  // vectors per fast-loop iteration
    const int64_t nfull = V / VW;                           // vectors holding VW tokens
    const int64_t vend = VEC ? min(v1, nfull) : v0;
    const int64_t n_it = vend > v0 ? (vend - v0) / STEP : 0;
    SlowState st{L};
    int64_t base = v0;
    if (n_it > 0) {
        const float shift = BLK ? bk.shift() : 0.f;
        const float seed = seed_theta<DT, BLK>(row, v0, c, key, ctx, pos, st.L.k, bk);
        st.L.bound(seed, shift);
        if (slot != nullptr && (threadIdx.x & 31) == 0 && seed < kInf) atomicMax(slot, bound_enc(seed));
        int64_t it = 0;
        int qn = 0;
        while (it < n_it) {
            RowPhilox rp;
            rp.init(key, ctx, pos);
            float tfa = st.L.tf;
            it = fast_scan<DT, VF, U>(rp, row, v0, it, n_it, c, st.L.tz, q, qn, slot, shift, tfa);
            st.L.bound(tfa, shift);
            if (qn > 0) st = flush_queue<DT, BLK>(st, q, qn, row, c, key, ctx, pos, bk, slot);
            qn = 0;
        }
        base = v0 + n_it * STEP;
    }
    if (base < v1) st = tail_loop<DT, BLK>(st, row, V, base, v1, c, key, ctx, pos, -kInf, bk, slot);
    L = st.L;
}

// ---------------------------------------------------------------- finalize

template <int DT>
__device__ __forceinline__ float logit_at(const RaceArgs& a, int64_t r, int64_t i) {
    const char* base = reinterpret_cast<const char*>(a.logits) + (size_t)r * (size_t)a.stride * (DT == 1 ? 2 : 4);
    return load_logit<DT>(base, i);
}

// Where the finishing steps read the logits of a row's listed tokens: the
// dense row in HBM (the streaming kernels), or the table of the row's
// candidates that the LM-head path keeps (its logits never reach HBM).
template <int DT>
struct DenseLogits {
    static constexpr bool kDense = true;
    const char* row;
    __device__ __forceinline__ float operator()(int64_t i) const { return load_logit<DT>(row, i); }
};
template <int DT>
__device__ __forceinline__ DenseLogits<DT> dense_logits(const RaceArgs& a, int64_t r) {
    return DenseLogits<DT>{reinterpret_cast<const char*>(a.logits) + (size_t)r * (size_t)a.stride * (DT == 1 ? 2 : 4)};
}

__device__ void walk_sequence(const RaceArgs& a, int s, int lane);

// Outputs of row r from its sorted entries: lane m holds the m-th smallest
// (key, token) of the row's list (dk fp64 when exact, sk fp32), nvalid of them
// usable.  Verify rows: the winner and its word.  Draft rows: the list, its
// multiplicities and labels (IID: the kr smallest multi-arrival scores).
template <int DT, bool VERIFY, class LP>
__device__ __forceinline__ void emit_row(const RaceArgs& a, int64_t r, double dk, float sk, int li, int nvalid, int kr,
                                         int lane, uint64_t key, uint64_t ctx, uint32_t pos, const LP& lp) {
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
    if (a.iid && kr <= 8) {
        // The same samples with the kr x kr candidates laid out at once: arrival j = e + 1 of
        // token t (its t-th list entry) sits in lane 8 (t mod 4) + e of slot t / 4.  Each lane
        // forms its arrival time, the 8-lane group its cumulative sums in arrival order (a
        // chain of shuffles, so G_{t,j} is summed exactly as the one-at-a-time version sums
        // it) and its scores; kr rounds of a warp argmin over (score, token, arrival) then
        // give the samples.  A token's later arrivals order after its earlier ones, so the
        // global kr smallest are the samples the one-at-a-time version finds.
        mult = 0;
        sample = -1;
        double h2[2];
        int t2[2], j2[2];
#pragma unroll
        for (int sl = 0; sl < 2; ++sl) {
            const int t = 4 * sl + (lane >> 3), e = lane & 7;
            const int tt = __shfl_sync(FULL, li, t);
            const bool valid = t < nuse && e < kr;
            const double E = valid ? exp1_f64(word_of(key, ctx, pos, tt, e + 1)) : 0.0;
            double G = E;
#pragma unroll
            for (int st = 1; st < 8; ++st) {
                const double prev = __shfl_up_sync(FULL, G, 1);
                if (e == st) G = prev + E;
            }
            const double ld = valid ? (double)lp(tt) : 0.0;
            h2[sl] = valid ? log(G) - ld / (double)a.T : (double)INFINITY;
            t2[sl] = valid ? tt : INT_MAX;
            j2[sl] = e + 1;
        }
        for (int m = 0; m < kr; ++m) {
            const int ls = (h2[1] < h2[0] || (h2[1] == h2[0] && (t2[1] < t2[0] || (t2[1] == t2[0] && j2[1] < j2[0])))) ? 1 : 0;
            double bh = ls ? h2[1] : h2[0];
            int bt = ls ? t2[1] : t2[0], bj = ls ? j2[1] : j2[0], bo = 2 * lane + ls;
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                const double oh = __shfl_xor_sync(FULL, bh, off);
                const int ot = __shfl_xor_sync(FULL, bt, off);
                const int oj = __shfl_xor_sync(FULL, bj, off);
                const int oo = __shfl_xor_sync(FULL, bo, off);
                if (oh < bh || (oh == bh && (ot < bt || (ot == bt && oj < bj)))) {
                    bh = oh;
                    bt = ot;
                    bj = oj;
                    bo = oo;
                }
            }
            if (bt == INT_MAX) break;  // fewer usable tokens than samples
            if (lane == m) sample = bt;
            if (mine && tok == bt) ++mult;
            if ((bo >> 1) == lane) {
                if (bo & 1) h2[1] = (double)INFINITY, t2[1] = INT_MAX;
                else h2[0] = (double)INFINITY, t2[0] = INT_MAX;
            }
        }
    } else if (a.iid) {
        // multi-arrival scores ln(G_{t,j}) - l_t/T of the nuse tokens, j = 1..kr;
        // the kr smallest (ties by token, then arrival) are the samples
        mult = 0;
        sample = -1;
        float lt = mine ? lp(li) : 0.0f;
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
        if (a.out_mult) a.out_mult[o] = lane < kr ? mult : 0;
        if (a.out_samples) a.out_samples[o] = lane < kr ? sample : -1;
    }
    if (lane == 0 && a.out_nd) a.out_nd[r] = nd;
}

// IID rows whose first-arrival list has no near ties: the multi-arrival
// scores in fp32, in key32's units (log2 of the summed -log2 u terms, minus
// l c).  Each term errs by at most its transform's bound (kErrAbs, measured)
// plus lg2.approx's error, the sum of at most 32 terms adds 31 roundings and
// the outer lg2.approx its error again, so every score is within
// key_err_bound + kBlkErr of its exact value (the derivation of kBlkErr covers
// this sum too).  When every gap between consecutive selected scores, and
// between the last selected and the best unselected one, exceeds the two
// bounds, the samples and their order are those of the exact scores and the
// row is written here; otherwise it returns false and the caller re-keys the
// row in fp64 (emit_row).
template <int DT, class LP>
__device__ __noinline__ bool iid_fast(const RaceArgs& a, int64_t r, float lk, int li, int nvalid, int kr, int lane,
                                      uint64_t key, uint64_t ctx, uint32_t pos, const LP lp) {
    const int nuse = min(nvalid, kr);
    const bool mine = lane < nuse;
    const int tok = mine ? li : -1;
    const float lt = mine ? lp(li) : 0.0f;
    float y = mine ? neg_log2_u(word_of(key, ctx, pos, li, 1)) : 0.0f;
    float h = mine ? lk : kInf;  // arrival 1's score is the list key itself
    // every lane's second arrival up front (independent chains); the rounds below then
    // extend a dependent chain only for third and later arrivals
    float y2 = 0.0f, h2 = kInf;
    if (kr > 1 && mine) {
        y2 = y + neg_log2_u(word_of(key, ctx, pos, tok, 2));
        h2 = fmaf(-lt, a.c, lg2_approx(y2));
    }
    int j = 1, mult = 0, sample = -1, nsel = 0;
    float selh = kInf;
    for (int m = 0; m < kr; ++m) {
        // warp argmin of (h, tok): each lane holds a distinct token, so the
        // winner's lane is the one holding bt
        float bh;
        const int bt = warp_argmin(h, mine ? tok : INT_MAX, bh);
        if (bt == INT_MAX) break;  // fewer usable tokens than samples
        if (lane == m) {
            sample = bt;
            selh = bh;
        }
        ++nsel;
        if (mine && tok == bt) {
            ++mult;
            ++j;
            if (j == 2 && j <= kr) {
                y = y2;
                h = h2;
            } else if (j <= kr) {
                y += neg_log2_u(word_of(key, ctx, pos, tok, j));
                h = fmaf(-lt, a.c, lg2_approx(y));
            } else {
                h = kInf;
            }
        }
    }
    float nxt = h;  // the best unselected score
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) nxt = fminf(nxt, __shfl_xor_sync(FULL, nxt, off));
    const float after = __shfl_down_sync(FULL, selh, 1);
    const float b = lane + 1 < nsel ? after : nxt;
    const bool bad = lane < nsel && b < kInf &&
                     !(b - selh > key_err_bound(selh) + key_err_bound(b) + 2.0f * kBlkErr);
    if (__any_sync(FULL, bad)) return false;
    const int nd = __popc(__ballot_sync(FULL, mult > 0));
    const int K = a.K;
    if (lane < K) {
        const size_t o = (size_t)r * K + lane;
        a.out_tok[o] = lane < kr ? tok : -1;
        if (a.out_key) a.out_key[o] = (mine && lane < kr) ? key_to_s(lk) : kInf;
        if (a.out_mult) a.out_mult[o] = lane < kr ? mult : 0;
        if (a.out_samples) a.out_samples[o] = lane < kr ? sample : -1;
    }
    if (lane == 0 && a.out_nd) a.out_nd[r] = nd;
    return true;
}

// Exact finish of a row whose list could not prove itself complete: tokens
// crowd its k-th key tau within the error bounds and the 32-entry list has no
// room left to hold them (always the case for k = 32 on a full list).  One
// more pass over the row collects every token whose list key is at most
// filter_slack(tau) (plus the block error) into shared memory, up to
// kRescanCap of them; the k smallest by their fp64 keys, in order, go to
// lanes 0..: (dk, li).  Every token whose exact key is at most the row's
// exact k-th key has a list key within that cut.  Returns false when more
// tokens than the buffer holds crowd the cut.  `scratch` holds
// 1 + 2 kRescanCap words.
constexpr int kRescanCap = 96;

template <int DT, bool BLK>
__device__ __noinline__ bool rescan_row(const RaceArgs& a, int64_t r, float tau, int kr, int lane, Blk bk,
                                        uint32_t* scratch, double& dk, int& li, int& nvalid) {
    constexpr int VW = DT == 1 ? 8 : 4;
    const uint64_t key = a.key[r], ctx = a.ctx[r];
    const uint32_t pos = a.pos[r];
    const char* row = reinterpret_cast<const char*>(a.logits) + (size_t)r * (size_t)a.stride * (DT == 1 ? 2 : 4);
    const float c = a.c;
    const float cut = filter_slack(tau) + (BLK ? 4.0f * kBlkErr : 0.f);
    const float tz = filter_tz(cut + (BLK ? bk.shift() : 0.f));
    int* cnt = reinterpret_cast<int*>(scratch);
    float* ck = reinterpret_cast<float*>(scratch + 1);
    int* ci = reinterpret_cast<int*>(scratch + 1 + kRescanCap);
    if (lane == 0) *cnt = 0;
    __syncwarp();
    RowPhilox rp;
    rp.init(key, ctx, pos);
    for (int64_t v0 = 0; v0 < a.nv; v0 += 32) {
        const int64_t v = v0 + lane;
        if (v < a.nv) {
            const uint4 dv = load_scalar<DT>(row, v, a.V);
            const uint4 d[2] = {dv, dv};
#pragma unroll
            for (int h = 0; h < (DT == 1 ? 2 : 1); ++h) {
                float l[4];
                block_logits<DT>(d, h, l);
                const uint32_t cb = DT == 1 ? (uint32_t)(2 * v + h) : (uint32_t)v;
                const uint4 q = rp.block(cb);
                const uint32_t wq[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int64_t i = (int64_t)4 * cb + e;
                    if (i < a.V && v * VW + 4 * h + e < a.V && filter_pass(wq[e], l[e], c, tz)) {
                        float k;
                        if constexpr (BLK)
                            k = block_key_of(key, ctx, pos, i, wq[e], l[e], c, bk.b, bk.B, bk.invB());
                        else
                            k = key32(wq[e], l[e], c);
                        if (k <= cut) {
                            const int slot = atomicAdd(cnt, 1);
                            if (slot < kRescanCap) {
                                ck[slot] = k;
                                ci[slot] = (int)i;
                            }
                        }
                    }
                }
            }
        }
    }
    __syncwarp();
    const int n = *cnt;
    if (n > kRescanCap) return false;
    // fp64 keys of the candidates (lane m holds candidates m, m + 32, m + 64)
    double d[3];
    int id[3];
#pragma unroll
    for (int t = 0; t < 3; ++t) {
        const int m = lane + 32 * t;
        d[t] = (double)INFINITY;
        id[t] = INT_MAX;
        if (m < n) {
            id[t] = ci[m];
            const uint32_t w = word_of(key, ctx, pos, id[t], 1);
            const float l = logit_at<DT>(a, r, id[t]);
            if constexpr (BLK) {
                uint32_t wf;
                const int J = block_words(key, ctx, pos, id[t], bk.b, bk.B, wf);
                d[t] = block_key64(w, J, wf, bk.b, bk.B, l, a.T);
            } else {
                d[t] = key64(w, l, a.T);
            }
        }
    }
    // the min(n, 32) smallest in order: lane m receives the m-th
    dk = (double)INFINITY;
    li = INT_MAX;
    const int take = min(n, 32);
    for (int m = 0; m < take; ++m) {
        double bd = d[0];
        int bi = id[0], bt = 0;
#pragma unroll
        for (int t = 1; t < 3; ++t)
            if (lex_less_d(d[t], id[t], bd, bi)) {
                bd = d[t];
                bi = id[t];
                bt = t;
            }
        double wd = bd;
        int wi = bi, wl = lane;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            const double od = __shfl_xor_sync(FULL, wd, off);
            const int oi = __shfl_xor_sync(FULL, wi, off);
            const int ol = __shfl_xor_sync(FULL, wl, off);
            if (lex_less_d(od, oi, wd, wi)) {
                wd = od;
                wi = oi;
                wl = ol;
            }
        }
        if (lane == m) {
            dk = wd;
            li = wi;
        }
        if (lane == wl) {
#pragma unroll
            for (int t = 0; t < 3; ++t)
                if (t == bt) {
                    d[t] = (double)INFINITY;
                    id[t] = INT_MAX;
                }
        }
    }
    nvalid = take;
    (void)kr;
    return true;
}

// Warp 0 finishes row r from its complete list (lk, li) and the drop bound.
// BLK: the near-tie keys are those of the row's block arrivals.
template <int DT, bool VERIFY, bool BLK, class LP>
__device__ __forceinline__ void finalize_row_lp(const RaceArgs& a, int64_t r, float lk, int li, float theta_drop,
                                                int kr, int kp, int lane, const LP& lp, Blk bk, uint32_t* scratch) {
    const int nvalid = __popc(__ballot_sync(FULL, lane < kp && lk < kInf));
    const float tau = nvalid >= kr ? __shfl_sync(FULL, lk, kr - 1) : kInf;
    // list-key error bound (block rows: widened by kBlkErr)
    auto err = [&](float k) { return BLK ? key_err_bound(k) + kBlkErr : key_err_bound(k); };
    bool complete;
    if (nvalid < kr)
        complete = theta_drop == kInf;
    else if (tau == -kInf)
        complete = true;
    else
        complete = theta_drop == kInf || theta_drop > tau + err(tau) + err(theta_drop);
    if (LP::kDense && !complete && nvalid >= kr && scratch != nullptr) {
        // the boundary is crowded: finish the row exactly with one more pass
        double dkr;
        int lir, nvr;
        if (rescan_row<DT, BLK>(a, r, tau, kr, lane, bk, scratch, dkr, lir, nvr)) {
            if (lane == 0 && a.status && tau > -kInf && fabsf(tau) > 65536.0f) atomicOr(a.status, PPS_FLAG_LOGIT_RANGE);
            emit_row<DT, VERIFY>(a, r, dkr, (float)dkr, lir, nvr, kr, lane, a.key[r], a.ctx[r], a.pos[r], lp);
            return;
        }
    }
    if (lane == 0 && a.status) {
        unsigned f = complete ? 0u : PPS_FLAG_GUARD;
        if (nvalid >= kr && tau > -kInf && fabsf(tau) > 65536.0f) f |= PPS_FLAG_LOGIT_RANGE;
        if (f) atomicOr(a.status, f);
    }
    // near ties among the first min(nvalid, kr+1) entries
    float nk = __shfl_down_sync(FULL, lk, 1);
    int lim = min(nvalid, kr + 1);
    bool close = lane + 1 < lim && !(nk - lk > err(lk) + err(nk));
    const bool any_close = __ballot_sync(FULL, close) != 0;
    const uint64_t key = a.key[r], ctx = a.ctx[r];
    const uint32_t pos = a.pos[r];
    if constexpr (!VERIFY && !BLK) {
        if (a.iid && !any_close && PPS_IID_FAST && iid_fast<DT>(a, r, lk, li, nvalid, kr, lane, key, ctx, pos, lp))
            return;
    }
    const bool need_exact = any_close || (!VERIFY && a.iid);
    double dk = (double)INFINITY;
    float sk = key_to_s(lk);
    if (need_exact) {
        if (lane < nvalid) {
            uint32_t w = word_of(key, ctx, pos, li, 1);
            if constexpr (BLK) {
                uint32_t wf;
                const int J = block_words(key, ctx, pos, li, bk.b, bk.B, wf);
                dk = block_key64(w, J, wf, bk.b, bk.B, lp(li), a.T);
            } else
                dk = key64(w, lp(li), a.T);
        }
        warp_sort_d(dk, li, lane);
        sk = (float)dk;
    }
    emit_row<DT, VERIFY>(a, r, dk, sk, li, nvalid, kr, lane, key, ctx, pos, lp);
}

// Warp 0 finishes row r of a streamed logits matrix from its complete list.
template <int DT, bool VERIFY, bool BLK = false>
__device__ __noinline__ void finalize_row(const RaceArgs& a, int64_t r, float lk, int li, float theta_drop, int kr,
                                          int kp, int lane, Blk bk = Blk{}, uint32_t* scratch = nullptr) {
    finalize_row_lp<DT, VERIFY, BLK>(a, r, lk, li, theta_drop, kr, kp, lane, dense_logits<DT>(a, r), bk, scratch);
}

// vectors per unit of the streaming kernel's row partition (see race_kernel)
__host__ __device__ constexpr int64_t race_unit(int dt) { return dt == 1 ? 32 * PPS_UNITS_VERIFY : 1; }

__device__ __forceinline__ int64_t warp_of(int64_t g, int64_t total, int64_t NW) {
    // largest w with floor(w*total/NW) <= g
    return ((g + 1) * NW - 1) / total;
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

// The walk of sequence s by the whole warp: per step one round of loads for
// the node (winner, word, draft row) and one for its draft list and children
// (lane m takes list slot m); emitted token t is kept by lane t % 32, and the
// scores of all emitted tokens are computed at once at the end.
__device__ __noinline__ void walk_sequence(const RaceArgs& a, int s, int lane) {
    const int W = a.gamma + 1;
    int c = __ldg(a.seq_off + s);
    if (c < 0 || c >= a.n_rows) {
        // no root row: nothing emitted, and the caller learns of it through the status word
        for (int t = lane; t < W; t += 32) {
            a.out_em[(size_t)s * W + t] = -1;
            a.out_sc[(size_t)s * W + t] = 0.0f;
        }
        if (lane == 0) {
            a.out_acc[s] = 0;
            a.out_ne[s] = 0;
            a.out_ss[s] = 0.0;
            if (a.status) atomicOr(a.status, PPS_FLAG_TREE);
        }
        return;
    }
    int acc = 0, ne = 0;
    int y_[3] = {-1, -1, -1};
    uint32_t w_[3] = {0u, 0u, 0u};
    auto keep = [&](int y, uint32_t w) {
        if ((ne & 31) == lane) {
            const int q = ne >> 5;
            if (q == 0) { y_[0] = y; w_[0] = w; }
            else if (q == 1) { y_[1] = y; w_[1] = w; }
            else { y_[2] = y; w_[2] = w; }
        }
        ++ne;
    };
    bool stopped = false;
    for (int step = 0; step < a.gamma; ++step) {
        const int y = __ldcg(a.out_winner + c);
        const uint32_t w = __ldcg(a.out_word + c);
        const int dr = __ldg(a.node_draft_row + c);
        if (y < 0) {
            stopped = true;
            break;
        }
        keep(y, w);
        int found = -1, nxt = -1;
        if (dr >= 0 && dr < a.n_draft) {
            const int nd = min(__ldg(a.draft_nd + dr), a.Kd);
            int t = -1, ch = -1;
            if (lane < nd) {
                t = __ldg(a.draft_tok + (size_t)dr * a.Kd + lane);
                ch = __ldg(a.child_node + (size_t)dr * a.Kd + lane);
            }
            const unsigned hit = __ballot_sync(FULL, lane < nd && t == y);
            if (hit) {
                found = __ffs(hit) - 1;
                nxt = __shfl_sync(FULL, ch, found);
            }
        }
        if (found < 0 || nxt < 0 || nxt >= a.n_rows) {
            stopped = true;
            break;
        }
        c = nxt;
        ++acc;
    }
    if (!stopped) {
        const int y = __ldcg(a.out_winner + c);
        const uint32_t w = __ldcg(a.out_word + c);
        if (y >= 0) keep(y, w);
    }
    // scores of the emitted tokens, their sum in emission order
    double A[3];
    double S = 0.0;
#pragma unroll
    for (int q = 0; q < 3; ++q) {
        const int t = q * 32 + lane;
        A[q] = t < ne ? score64(w_[q]) : 0.0;
        if (t < W) {
            a.out_em[(size_t)s * W + t] = t < ne ? y_[q] : -1;
            a.out_sc[(size_t)s * W + t] = (float)A[q];
        }
    }
    for (int t = 0; t < ne; ++t) {
        const int q = t >> 5;
        S += __shfl_sync(FULL, q == 0 ? A[0] : (q == 1 ? A[1] : A[2]), t & 31);
    }
    if (lane == 0) {
        a.out_acc[s] = acc;
        a.out_ne[s] = ne;
        a.out_ss[s] = S;
    }
}

// End of a row segment: publish the warp's list, or merge the row's lists if
// this warp is the last to finish the row, then finish the row (and the walk
// of its sequence when it is the sequence's last node).  Out of line.
// Sequence ticket after node row r is final: the warp that finishes a
// sequence's last node walks it.
__device__ __noinline__ void sequence_ticket(const RaceArgs& a, int64_t r, int lane) {
    __threadfence();
    int s = 0;
    unsigned last = 0;
    if (lane == 0) {
        s = seq_of_node(a.seq_off, a.n_seq, r);
        int nn = __ldg(a.seq_off + s + 1) - __ldg(a.seq_off + s);
        unsigned t = atomicAdd(a.seq_cnt + s, 1u);
        last = t == (unsigned)(nn - 1);
        if (last) a.seq_cnt[s] = 0u;
    }
    if (__shfl_sync(FULL, last, 0)) {
        __threadfence();
        walk_sequence(a, __shfl_sync(FULL, s, 0), lane);
    }
    __syncwarp();
}

// Merge the partial lists of warps first_w..last_w of row r into (lk, li) and
// lower theta_drop to a bound on every key the merged list leaves out.  The
// partials were written by warps all over the GPU (L2 round trips of a
// microsecond or so), so they are loaded kMergeBatch at a time, all loads of a
// batch in flight together, and a batch is merged as a tree (independent pairs
// first), so that a small launch with many warps per row does not pay one
// round trip and one dependent merge per partial.  Merging two sorted lists
// keeps the kp smallest of their union and reports the smallest key it drops,
// so every key left out of the result is >= the minimum of both lists' drop
// bounds and the dropped keys.
constexpr int kMergeBatch = 8;

__device__ __forceinline__ void merge_partials(const RaceArgs& a, int64_t r, int64_t first_w, int64_t last_w, int kp,
                                               int lane, float& lk, int& li, float& theta_drop) {
    for (int64_t w0 = first_w; w0 <= last_w; w0 += kMergeBatch) {
        const int nb = (int)min((int64_t)kMergeBatch, last_w - w0 + 1);  // warp-uniform
        float pk[kMergeBatch], pd[kMergeBatch];
        int pi[kMergeBatch];
#pragma unroll
        for (int b = 0; b < kMergeBatch; ++b) {
            pk[b] = kInf;
            pi[b] = INT_MAX;
            pd[b] = kInf;
            if (b < nb) {
                const Partial* Q = a.partials + (w0 + b + r);
                pk[b] = __ldcg(Q->key + lane);
                pi[b] = __ldcg(Q->idx + lane);
                pd[b] = __ldcg(&Q->theta_drop);
            }
        }
        // tree: (0,1) (2,3) (4,5) (6,7), then (0,2) (4,6), then (0,4); empty lists are skipped
#pragma unroll
        for (int s = 1; s < kMergeBatch; s <<= 1) {
#pragma unroll
            for (int b = 0; b + s < kMergeBatch; b += 2 * s) {
                if (b + s < nb) {
                    const float dk = warp_merge<true>(pk[b], pi[b], pk[b + s], pi[b + s], kp, lane);
                    pd[b] = fminf(fminf(pd[b], pd[b + s]), dk);
                }
            }
        }
        const float dk = warp_merge<true>(lk, li, pk[0], pi[0], kp, lane);
        theta_drop = fminf(theta_drop, fminf(pd[0], dk));
    }
}

// Merge by selection rounds, for at most 32 partial lists: list j is staged in
// row j of s_k / s_i (entry e at [j * 32 + e], e < kp) by asynchronous 16-byte
// copies that every lane issues for its whole list before one wait (one L2
// round trip for the lot), lane j holds the head of list j, and each of kp
// rounds moves the warp's smallest head (key, token) to entry m of the merged
// list and advances its lane.  One warp argmin per output entry replaces one
// dependent bitonic merge per list.  Tokens are unique across the lists
// (disjoint segments of one row), so only the owner's head matches the
// winner.  The smallest head left over is the smallest listed key dropped.
// s_k and s_i are 16-byte aligned.
__device__ __forceinline__ void copy16_async(void* smem, const void* gmem) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(smem)),
                 "l"(gmem)
                 : "memory");
}

__device__ __noinline__ void merge_rounds(const RaceArgs& a, int64_t r, int64_t first_w, int P, int kp, int lane,
                                          float* s_k, int* s_i, float& lk, int& li, float& theta_drop) {
    float th = kInf;
    if (lane < P) {
        const Partial* Q = a.partials + (first_w + lane + r);
        th = __ldcg(&Q->theta_drop);
        for (int e = 0; e < kp; e += 4) {
            copy16_async(s_k + lane * 32 + e, Q->key + e);
            copy16_async(s_i + lane * 32 + e, Q->idx + e);
        }
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
    __syncwarp();
    int h = 0;
    float hk = lane < P ? s_k[lane * 32] : kInf;
    int hi = lane < P ? s_i[lane * 32] : INT_MAX;
    lk = kInf;
    li = INT_MAX;
    for (int m = 0; m < kp; ++m) {
        float bk;
        const int bi = warp_argmin(hk, hi, bk);
        if (bi == INT_MAX) break;  // fewer listed entries than kp (warp-uniform)
        if (lane == m) {
            lk = bk;
            li = bi;
        }
        if (hi == bi) {
            ++h;
            hk = h < kp ? s_k[lane * 32 + h] : kInf;
            hi = h < kp ? s_i[lane * 32 + h] : INT_MAX;
        }
    }
    float d = fminf(hk, th);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) d = fminf(d, __shfl_xor_sync(FULL, d, o));
    theta_drop = fminf(theta_drop, d);
    __syncwarp();
}

template <int DT, bool VERIFY, bool BLK>
__device__ __noinline__ void finish_segment(const RaceArgs& a, int64_t r, int64_t gw, int64_t NW, int64_t nb,
                                            int64_t v0, int64_t v1, const WarpList L, int kr, int kp, Blk bk,
                                            uint32_t* scratch, float* s_mk, int* s_mi) {
    const int lane = threadIdx.x & 31;
    const int64_t nv = a.nv;
    float lk = L.lk;
    int li = L.li;
    // every token of the segment left out of the list has a key >= theta_drop
    float theta_drop = L.drop();
    bool final_here = v0 == 0 && v1 == nv;
    if (!final_here) {
        // publish this segment's list; the last warp of the row merges all segments
        Partial* P = a.partials + (gw + r);
        P->key[lane] = lk;
        P->idx[lane] = li;
        if (lane == 0) P->theta_drop = theta_drop;
        __threadfence();
        __syncwarp();
        const int64_t units = a.n_rows * nb;
        const int64_t first_w = warp_of(r * nb, units, NW);
        const int64_t last_w = warp_of(r * nb + nb - 1, units, NW);
        unsigned last = 0;
        if (lane == 0) {
            unsigned t = atomicAdd(a.row_cnt + r, 1u);
            last = t == (unsigned)(last_w - first_w);
            if (last) {
                a.row_cnt[r] = 0u;
                if (a.row_bound) a.row_bound[r] = 0u;
            }
        }
        final_here = __shfl_sync(FULL, last, 0) != 0;
        if (final_here) {
            __threadfence();
            lk = kInf;
            li = INT_MAX;
            theta_drop = kInf;
            if (last_w - first_w < 32)
                merge_rounds(a, r, first_w, (int)(last_w - first_w + 1), kp, lane, s_mk, s_mi, lk, li, theta_drop);
            else
                merge_partials(a, r, first_w, last_w, kp, lane, lk, li, theta_drop);
        }
    }
    if (final_here) {
        finalize_row<DT, VERIFY, BLK>(a, r, lk, li, theta_drop, kr, kp, lane, bk, scratch);
        if constexpr (VERIFY) sequence_ticket(a, r, lane);
    }
}

// ---------------------------------------------------------------- the kernel
//
// Every warp is an independent worker.  A row is cut into nb units of
// race_unit(DT) vectors (the last may be shorter), and warp gw of NW streams the
// units [gw*U/NW, (gw+1)*U/NW) of the U = n_rows * nb units in row order.  For
// bf16 rows a unit is one fast-loop iteration, so that a segment ends on an
// iteration boundary and only a row's ragged end takes the scalar tail
// (measured on the bench tree: verify 0.282 -> 0.272 ms, draft 0.248 ->
// 0.235 ms); fp32 rows keep units of one vector (iteration units made the
// fp32 tree slower, 7.35 -> 7.73 ms).  A row cut between warps is merged and finished by
// the warp that arrives last at the row's counter; a sequence's walk is run by
// the warp that finishes its last node.  No warp ever waits for another and
// the kernel has no block-wide barrier.

template <int DT, bool VERIFY, bool VEC, bool BLK>
__global__ void __launch_bounds__(kThreads, BLK ? PPS_BLOCK_MIN_BLOCKS : PPS_RACE_MIN_BLOCKS) race_kernel(const RaceArgs a) {
    __shared__ uint32_t s_queue[kQueueCap];
    __shared__ __align__(16) float s_mk[32 * 32];  // staging of the partial lists merged by merge_rounds
    __shared__ __align__(16) int s_mi[32 * 32];
    pdl_wait();  // the previous kernel's outputs (row ids, lists) and the workspace it used
    pdl_launch_dependents();
    const int64_t NW = a.G;
    const int64_t gw = blockIdx.x;
    const float c = a.c;
    const int64_t nv = a.nv;
    const size_t esz = DT == 1 ? 2 : 4;
    constexpr int64_t kUnit = race_unit(DT);
    const int64_t nb = (nv + kUnit - 1) / kUnit;
    const int64_t units = a.n_rows * nb;
    const int64_t u0 = gw * units / NW, u1 = (gw + 1) * units / NW;

    for (int64_t r = u0 / nb; u0 < u1 && r < a.n_rows && r * nb < u1; ++r) {
        const int64_t v0 = (max(u0, r * nb) - r * nb) * kUnit;
        const int64_t v1 = min((min(u1, (r + 1) * nb) - r * nb) * kUnit, nv);
        int kr = 1;
        if (!VERIFY) {
            kr = a.row_k ? __ldg(a.row_k + r) : a.K;
            kr = max(1, min(kr, a.K));
        }
        const int kp = min(32, 2 * kr + 1);
        const uint64_t key = __ldg(a.key + r), ctx = __ldg(a.ctx + r);
        const uint32_t pos = __ldg(a.pos + r);
        const char* row = reinterpret_cast<const char*>(a.logits) + (size_t)r * (size_t)a.stride * esz;

        Blk bk;
        if constexpr (BLK) {
            bk.b = __ldg(a.row_block + r);
            bk.B = a.n_blocks;
        }
        WarpList L;
        L.reset(kp, kr);
        // A one-token draft list is a target race, and a list of a few tokens is close to one:
        // such rows stream like verify rows (one filter test per vector; measured: lists of up
        // to 4 gain, lists of 8 lose).  A row cut between warps shares its filter bound (verify,
        // short-list draft and proposal rows: on longer lists the shared bound saves too little).
        const bool one = VERIFY || (!BLK && kr <= PPS_VF_MAXK);
        uint32_t* slot = nullptr;
        if constexpr (PPS_ROWBOUND)
            if ((one || BLK) && a.row_bound && (v0 > 0 || v1 < nv)) slot = a.row_bound + r;
        if (!VERIFY && !BLK && one)
            stream_segment<DT, VEC, false, true, PPS_UNITS_VERIFY>(L, row, a.V, v0, v1, c, key, ctx, pos, s_queue,
                                                                 bk, slot);
        else
            stream_segment<DT, VEC, BLK, VERIFY || DT == 0, VERIFY ? PPS_UNITS_VERIFY : PPS_UNITS>(
                L, row, a.V, v0, v1, c, key, ctx, pos, s_queue, bk, slot);

        finish_segment<DT, VERIFY, BLK>(a, r, gw, NW, nb, v0, v1, L, kr, kp, bk, s_queue, s_mk, s_mi);
    }
}


#include "pps_trunc.cuh"
#include "pps_lmhead.cuh"

// the race kernel instance: dtype x (verify | block draft | draft) x vec
static const void* race_fn(int dtype, bool verify, bool blk, bool vec) {
    if (dtype == 1) {
        if (verify) return vec ? (const void*)race_kernel<1, true, true, false> : (const void*)race_kernel<1, true, false, false>;
        if (blk) return vec ? (const void*)race_kernel<1, false, true, true> : (const void*)race_kernel<1, false, false, true>;
        return vec ? (const void*)race_kernel<1, false, true, false> : (const void*)race_kernel<1, false, false, false>;
    }
    if (verify) return vec ? (const void*)race_kernel<0, true, true, false> : (const void*)race_kernel<0, true, false, false>;
    if (blk) return vec ? (const void*)race_kernel<0, false, true, true> : (const void*)race_kernel<0, false, false, true>;
    return vec ? (const void*)race_kernel<0, false, true, false> : (const void*)race_kernel<0, false, false, false>;
}

int race_grid(int64_t total, int dtype, bool verify, bool vec, bool blk, int64_t n_rows) {
    const int kind = verify ? 1 : (blk ? 2 : 0);
    const int o = resident_ctas(kOccRace + (dtype * 3 + kind) * 2 + (vec ? 1 : 0),
                                race_fn(dtype, verify, blk && !verify, vec), kThreads);
    int64_t g = (int64_t)device_sm_count() * o;
    int64_t by_size = (total + kMinVecsPerWarp - 1) / kMinVecsPerWarp;
    if (by_size < g) g = by_size;
    if (PPS_SEG_CAP > 0 && n_rows > 0 && n_rows * PPS_SEG_CAP < g) g = n_rows * PPS_SEG_CAP;
    if (n_rows > 0) {
        // every warp gets at least one unit (one fast iteration of a row), so every
        // warp a row's counter waits for streams part of it
        const int64_t unit = race_unit(dtype);
        const int64_t units = n_rows * ((total / n_rows + unit - 1) / unit);
        if (units < g) g = units;
    }
    if (g > kGridMax) g = kGridMax;
    if (g < 1) g = 1;
    return (int)g;
}

cudaError_t launch_race(const RaceArgs& a, int dtype, bool verify, bool vec, cudaStream_t stream) {
    dim3 grid(a.G), block(kThreads);
    cudaError_t e = cudaSuccess;
    const bool blk = !verify && a.row_block != nullptr;
    if (dtype == 1) {
        if (verify) {
            if (vec) e = launch_pdl(race_kernel<1, true, true, false>, grid, block, 0, stream, a);
            else e = launch_pdl(race_kernel<1, true, false, false>, grid, block, 0, stream, a);
        } else if (blk) {
            if (vec) e = launch_pdl(race_kernel<1, false, true, true>, grid, block, 0, stream, a);
            else e = launch_pdl(race_kernel<1, false, false, true>, grid, block, 0, stream, a);
        } else {
            if (vec) e = launch_pdl(race_kernel<1, false, true, false>, grid, block, 0, stream, a);
            else e = launch_pdl(race_kernel<1, false, false, false>, grid, block, 0, stream, a);
        }
    } else {
        if (verify) {
            if (vec) e = launch_pdl(race_kernel<0, true, true, false>, grid, block, 0, stream, a);
            else e = launch_pdl(race_kernel<0, true, false, false>, grid, block, 0, stream, a);
        } else if (blk) {
            if (vec) e = launch_pdl(race_kernel<0, false, true, true>, grid, block, 0, stream, a);
            else e = launch_pdl(race_kernel<0, false, false, true>, grid, block, 0, stream, a);
        } else {
            if (vec) e = launch_pdl(race_kernel<0, false, true, false>, grid, block, 0, stream, a);
            else e = launch_pdl(race_kernel<0, false, false, false>, grid, block, 0, stream, a);
        }
    }
    return e != cudaSuccess ? e : cudaGetLastError();
}

// Rows stay whole where the grid allows (a segment's candidate count grows
// like k ln(segment / k), and a row finished by one warp needs no merge):
// with at most as many rows as resident warps, each row gets the same number
// of warps s; with more rows, the grid is the resident one.
static const void* trunc_fn(int dtype, bool verify, bool blk, bool vec) {
    if (dtype == 1) {
        if (verify) return vec ? (const void*)trunc_kernel<1, true, true, false> : (const void*)trunc_kernel<1, true, false, false>;
        if (blk) return vec ? (const void*)trunc_kernel<1, false, true, true> : (const void*)trunc_kernel<1, false, false, true>;
        return vec ? (const void*)trunc_kernel<1, false, true, false> : (const void*)trunc_kernel<1, false, false, false>;
    }
    if (verify) return vec ? (const void*)trunc_kernel<0, true, true, false> : (const void*)trunc_kernel<0, true, false, false>;
    if (blk) return vec ? (const void*)trunc_kernel<0, false, true, true> : (const void*)trunc_kernel<0, false, false, true>;
    return vec ? (const void*)trunc_kernel<0, false, true, false> : (const void*)trunc_kernel<0, false, false, false>;
}

int trunc_grid(int64_t total, int64_t n_rows, int dtype, bool verify, bool vec, bool blk) {
    const int kind = verify ? 1 : (blk ? 2 : 0);
    const int o = resident_ctas(kOccTrunc + (dtype * 3 + kind) * 2 + (vec ? 1 : 0),
                                trunc_fn(dtype, verify, blk && !verify, vec), kThreads);
    int64_t g = (int64_t)device_sm_count() * o;
    int64_t by_size = (total + kMinVecsPerWarp - 1) / kMinVecsPerWarp;
    if (by_size < g) g = by_size;
    if (n_rows > 0 && n_rows <= g) g = n_rows * (g / n_rows);
    if (g > kGridMax) g = kGridMax;
    if (g < 1) g = 1;
    return (int)g;
}

cudaError_t launch_trunc(const RaceArgs& a, int dtype, bool verify, bool vec, cudaStream_t stream) {
    dim3 grid(a.G), block(kThreads);
    cudaError_t e = cudaSuccess;
    const bool blk = !verify && a.row_block != nullptr;
    if (dtype == 1) {
        if (verify) {
            if (vec) e = launch_pdl(trunc_kernel<1, true, true, false>, grid, block, 0, stream, a);
            else e = launch_pdl(trunc_kernel<1, true, false, false>, grid, block, 0, stream, a);
        } else if (blk) {
            if (vec) e = launch_pdl(trunc_kernel<1, false, true, true>, grid, block, 0, stream, a);
            else e = launch_pdl(trunc_kernel<1, false, false, true>, grid, block, 0, stream, a);
        } else {
            if (vec) e = launch_pdl(trunc_kernel<1, false, true, false>, grid, block, 0, stream, a);
            else e = launch_pdl(trunc_kernel<1, false, false, false>, grid, block, 0, stream, a);
        }
    } else {
        if (verify) {
            if (vec) e = launch_pdl(trunc_kernel<0, true, true, false>, grid, block, 0, stream, a);
            else e = launch_pdl(trunc_kernel<0, true, false, false>, grid, block, 0, stream, a);
        } else if (blk) {
            if (vec) e = launch_pdl(trunc_kernel<0, false, true, true>, grid, block, 0, stream, a);
            else e = launch_pdl(trunc_kernel<0, false, false, true>, grid, block, 0, stream, a);
        } else {
            if (vec) e = launch_pdl(trunc_kernel<0, false, true, false>, grid, block, 0, stream, a);
            else e = launch_pdl(trunc_kernel<0, false, false, false>, grid, block, 0, stream, a);
        }
    }
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace pps
