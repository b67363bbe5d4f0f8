// pps_trunc.cuh -- the truncated race: top-k, then top-p, then the race over
// the surviving tokens.  Included by pps_race.cu, whose Philox, lists, row
// finalisation and tree walk it reuses (one translation unit).
//
// Truncation (the experiments sample with top-k = 50, top-p = 1, Sec. 6; a
// truncated distribution has a support of at most k tokens, Sec. 4.2) sets
// P = 0, i.e. E/P = +inf, outside the kept set S, so the race of the truncated
// distribution is argmin over S of s = ln E - l/T (the renormalisation of P on
// S does not move the argmin).  The set: every token whose logit is >= l_(k),
// the k-th largest usable logit (all ties of l_(k) are kept); then, if
// top_p < 1, whole groups of equal logits are removed in ascending order while
// the running probability mass (softmax(l/T) over the top-k set, summed token
// by token in ascending order) is <= 1 - top_p; the top group always stays.
//
// Work per row.  The streaming pass only finds S: one max of the iteration's
// logits per lane (packed bf16x2 max for bf16 rows) against the warp's
// threshold, the k-th entry of a per-warp top list of up to 64 (logit, token)
// entries.  No Philox word is needed for a token outside S, so the pass is
// bound by HBM rather than by the multiply pipe.  Vectors with a logit at or
// over the threshold are queued and their tokens merged into the list
// (bitonic sort and merges).  Tokens below the threshold are below l_(k) and
// can be dropped for good; a token evicted from a full list is recorded in
// `dropmax`, and if one ties with l_(k) the row's list does not hold the whole
// tie group: the row is then finished by a counting pass (for top-p) and, when
// the tie group stays in S, by the exact fp32 race of pps_race.cu over the
// tokens with logit >= l_(k).  Otherwise the finishing warp keys the <= 64
// surviving tokens with the race's fp32 key, keeps the 32 smallest and hands
// them to finalize_row with a drop bound of +inf (S is complete, nothing was
// dropped); finalize_row re-keys in fp64 (s = ln E - l/T) every pair closer
// than the fp32 error bounds, so the row is emitted exactly like the
// untruncated race.

#ifndef PPS_TRUNC_UNITS
#define PPS_TRUNC_UNITS 8  // 16-byte vectors per lane per iteration of the top-k scan (even)
#endif
#ifndef PPS_TRUNC_EAGER
#define PPS_TRUNC_EAGER 96  // buffered candidates at which a queue flush also compacts
#endif
#ifndef PPS_TRUNC_MIN_BLOCKS
#define PPS_TRUNC_MIN_BLOCKS 20
#endif

// ---------------------------------------------------------------- top lists
// A top list holds up to 64 entries (v, i) in "top order": logit descending,
// then token ascending.  Entry m sits in lane m (av, ai) for m < 32 and in
// lane m - 32 (bv, bi) otherwise; empty entries are (-inf, INT_MAX).  NaN and
// -inf logits never enter.

__device__ __forceinline__ bool top_before(float av, int ai, float bv, int bi) {
    return av > bv || (av == bv && ai < bi);
}

// bitonic sort of one entry per lane into top order (lane 0 first)
__device__ __forceinline__ void top_sort(float& v, int& i, int lane) {
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            const float ov = __shfl_xor_sync(FULL, v, stride);
            const int oi = __shfl_xor_sync(FULL, i, stride);
            const bool up = (lane & size) == 0 || size == 32;
            const bool lower = (lane & stride) == 0;
            const bool o_first = top_before(ov, oi, v, i);
            const bool take = (lower == up) ? o_first : (!o_first && !(ov == v && oi == i));
            if (take) {
                v = ov;
                i = oi;
            }
        }
    }
}

// bitonic half-cleaner pass over a bitonic sequence (one entry per lane)
__device__ __forceinline__ void top_clean(float& v, int& i, int lane) {
#pragma unroll
    for (int stride = 16; stride > 0; stride >>= 1) {
        const float ov = __shfl_xor_sync(FULL, v, stride);
        const int oi = __shfl_xor_sync(FULL, i, stride);
        const bool lower = (lane & stride) == 0;
        const bool o_first = top_before(ov, oi, v, i);
        if (lower ? o_first : (!o_first && !(ov == v && oi == i))) {
            v = ov;
            i = oi;
        }
    }
}

// two sorted lists x, y -> h = the first 32 of their union, l = the last 32, both sorted
__device__ __forceinline__ void top_merge(float xv, int xi, float yv, int yi, float& hv, int& hi, float& lv, int& li,
                                          int lane) {
    const float rv = __shfl_sync(FULL, yv, 31 - lane);
    const int ri = __shfl_sync(FULL, yi, 31 - lane);
    const bool xf = top_before(xv, xi, rv, ri);
    hv = xf ? xv : rv;
    hi = xf ? xi : ri;
    lv = xf ? rv : xv;
    li = xf ? ri : xi;
    top_clean(hv, hi, lane);
    top_clean(lv, li, lane);
}

struct TopList {
    float av, bv;   // entries lane and lane + 32
    int ai, bi;
    float thr;      // logit of entry k-1 (-inf while fewer than k entries): tokens below it cannot be in S
    float dropmax;  // largest logit evicted from the list (-inf: none)

    __device__ __forceinline__ void reset() {
        av = bv = -kInf;
        ai = bi = INT_MAX;
        thr = -kInf;
        dropmax = -kInf;
    }
    __device__ __forceinline__ float entry(int m) const {  // m warp-uniform
        const float x = __shfl_sync(FULL, av, m & 31), y = __shfl_sync(FULL, bv, m & 31);
        return m < 32 ? x : y;
    }
    // Merge a batch in top order (one entry per lane).  The first 32 of
    // (a, batch) are the new a; the rest merged with b gives the new b and
    // the evicted 32 (every entry of the old a precedes every entry of b, so
    // the first 64 of the union are exactly these).
    __device__ __forceinline__ void insert_sorted(float cv, int ci, int k, int lane) {
        float xh, xl, yh, yl;
        int xhi, xli, yhi, yli;
        top_merge(av, ai, cv, ci, xh, xhi, xl, xli, lane);
        top_merge(xl, xli, bv, bi, yh, yhi, yl, yli, lane);
        av = xh;
        ai = xhi;
        bv = yh;
        bi = yhi;
        dropmax = fmaxf(dropmax, __shfl_sync(FULL, yl, 0));
        thr = fmaxf(thr, entry(k - 1));
    }
    // insert one warp-uniform entry: find its place by ballots, shift the rest down
    __device__ __forceinline__ void insert_one(float cv, int ci, int k, int lane) {
        const int pos = __popc(__ballot_sync(FULL, top_before(av, ai, cv, ci))) +
                        __popc(__ballot_sync(FULL, top_before(bv, bi, cv, ci)));
        if (pos >= 2 * 32) {
            dropmax = fmaxf(dropmax, cv);
            return;
        }
        const float a31 = __shfl_sync(FULL, av, 31), b63 = __shfl_sync(FULL, bv, 31);
        const int a31i = __shfl_sync(FULL, ai, 31);
        float pa = __shfl_up_sync(FULL, av, 1), pb = __shfl_up_sync(FULL, bv, 1);
        int pai = __shfl_up_sync(FULL, ai, 1), pbi = __shfl_up_sync(FULL, bi, 1);
        if (lane == 0) {
            pb = a31;
            pbi = a31i;
        }
        if (lane > pos) {
            av = pa;
            ai = pai;
        } else if (lane == pos) {
            av = cv;
            ai = ci;
        }
        if (32 + lane > pos) {
            bv = pb;
            bi = pbi;
        } else if (32 + lane == pos) {
            bv = cv;
            bi = ci;
        }
        dropmax = fmaxf(dropmax, b63);
        thr = fmaxf(thr, entry(k - 1));
    }
    // A token can still change S: above the threshold, or tied with it while no
    // token of that logit has been evicted yet (once one has, the row's tie
    // group at that logit, if it is l_(k), overflows whatever else arrives).
    __device__ __forceinline__ bool wants(float x) const {
        return x > -kInf && (x > thr || (x == thr && dropmax < thr));
    }
    // one round: every lane offers (v, i) or nothing (-inf); few offers go in one
    // by one, more are sorted and merged
    __device__ __forceinline__ void offer(float v, int i, int k, int lane) {
        const unsigned vm = __ballot_sync(FULL, v > -kInf);
        if (__popc(vm) <= 2) {
            unsigned m = vm;
            while (m) {
                const int src = __ffs(m) - 1;
                m &= m - 1;
                insert_one(__shfl_sync(FULL, v, src), __shfl_sync(FULL, i, src), k, lane);
            }
        } else {
            if (v == -kInf) i = INT_MAX;
            top_sort(v, i, lane);
            insert_sorted(v, i, k, lane);
        }
    }
};

// Offer each lane's candidates (logits cv[e] of tokens ci[e]; -inf = none) to
// the list: every round the lanes' best remaining candidates at or over the
// threshold are sorted and merged; ends when no lane has one.
template <int N>
__device__ __forceinline__ void top_offer(TopList& L, float (&cv)[N], const int (&ci)[N], int k, int lane) {
    while (true) {
        float bv = -kInf;
        int bi = INT_MAX, be = -1;
#pragma unroll
        for (int e = 0; e < N; ++e) {
            if (L.wants(cv[e]) && top_before(cv[e], ci[e], bv, bi)) {
                bv = cv[e];
                bi = ci[e];
                be = e;
            }
        }
        if (__ballot_sync(FULL, be >= 0) == 0) break;
        L.offer(bv, bi, k, lane);
#pragma unroll
        for (int e = 0; e < N; ++e)
            if (e == be) cv[e] = -kInf;
    }
}

// ---------------------------------------------------------------- vector helpers

// any half of the bf16 pair m >= the bf16 pair t2 (NaN halves compare false)
__device__ __forceinline__ bool bf2_any_ge(uint32_t m, uint32_t t2) {
    uint32_t r;
    asm("{\n\t.reg .pred p, q;\n\t"
        "setp.ge.bf16x2 p|q, %1, %2;\n\t"
        "or.pred p, p, q;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(r)
        : "r"(m), "r"(t2));
    return r != 0;
}

// token e of a 16-byte vector as fp32 (exact)
template <int DT>
__device__ __forceinline__ float vec_token(const uint4& d, int e) {  // e a compile-time constant after unrolling
    const uint32_t w4[4] = {d.x, d.y, d.z, d.w};
    const uint32_t w = w4[DT == 1 ? e >> 1 : e];
    if constexpr (DT == 1) return (e & 1) ? bf16_hi(w) : bf16_lo(w);
    else return __uint_as_float(w);
}

// largest usable logit of vectors d[k0 .. k0+n) (NaN ignored, -inf if none)
template <int DT, int N>
__device__ __forceinline__ float vecs_max(const uint4 (&d)[N], int k0, int n) {
    float r = -kInf;
#pragma unroll
    for (int k = k0; k < k0 + n; ++k) {
        if constexpr (DT == 1) {
            const uint32_t m = bf2_max(bf2_max(d[k].x, d[k].y), bf2_max(d[k].z, d[k].w));
            r = fmaxf(r, fmaxf(bf16_lo(m), bf16_hi(m)));
        } else {
            r = fmaxf(r, fmaxf(fmaxf(__uint_as_float(d[k].x), __uint_as_float(d[k].y)),
                               fmaxf(__uint_as_float(d[k].z), __uint_as_float(d[k].w))));
        }
    }
    return r;  // fmaxf returns the non-NaN operand
}

// ---------------------------------------------------------------- the top-k scan

// order-preserving unsigned key of a float (NaN never reaches it)
__device__ __forceinline__ uint32_t order_key(float x) {
    const uint32_t b = __float_as_uint(x);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float from_order_key(uint32_t u) {
    return __uint_as_float((u & 0x80000000u) ? (u & 0x7fffffffu) : ~u);
}

// Threshold for an empty buffer, from the first iteration's vectors: the
// k-th largest of the 32 x NV per-vector maxima (bitwise search on order
// keys).  They are maxima of distinct vectors of the segment, so at least k
// of its tokens reach it and l_(k) >= it.
template <int DT>
__device__ __forceinline__ float seed_thr(const uint4 (&d)[PPS_TRUNC_UNITS], int k) {
    constexpr int NV = PPS_TRUNC_UNITS;
    uint32_t key[NV];
#pragma unroll
    for (int j = 0; j < NV; ++j) key[j] = order_key(vecs_max<DT>(d, j, 1));
    uint32_t res = 0;
    for (int b = 31; b >= 0; --b) {
        const uint32_t cand = res | (1u << b);
        int n = 0;
#pragma unroll
        for (int j = 0; j < NV; ++j) n += key[j] >= cand;
        if (__reduce_add_sync(FULL, (unsigned)n) >= (unsigned)k) res = cand;
    }
    return from_order_key(res);
}

// The scan appends every token the segment may still need to a per-warp
// buffer in shared memory and raises the threshold only when the buffer
// fills: then the k-th largest logit t of the buffer becomes the threshold
// and the buffer keeps the tokens above t and as many tied with t as the
// 64-entry list holds (dropmax records the rest).  Appending is cheap; the
// exact selection runs a few times per segment.
constexpr int kCandCap = 256;

struct CandState {
    float thr;      // lower bound of l_(k): tokens below it cannot be in S
    float dropmax;  // largest logit dropped from the buffer (-inf: none)
    int n;          // buffered entries
    // tokens that may still change S (see TopList::wants)
    __device__ __forceinline__ bool wants(float x) const {
        return x > -kInf && (x > thr || (x == thr && dropmax < thr));
    }
};

template <int DT>
__device__ __noinline__ CandState cand_compact(CandState C, float* sv, int* si, int k) {
    constexpr int PER = kCandCap / 32;
    const int lane = threadIdx.x & 31;
    if (C.n < k) return C;
    float v[PER];
    int ix[PER];
#pragma unroll
    for (int j = 0; j < PER; ++j) {
        const int q = j * 32 + lane;
        v[j] = q < C.n ? sv[q] : -kInf;
        ix[j] = q < C.n ? si[q] : INT_MAX;
    }
    __syncwarp();
    // t = the k-th largest buffered logit, bit by bit on order keys (bf16
    // values: the high 16 bits decide, the low ones are all 0 or all 1)
    uint32_t res = 0;
    for (int b = 31; b >= (DT == 1 ? 16 : 0); --b) {
        const uint32_t cand = res | (1u << b);
        int n = 0;
#pragma unroll
        for (int j = 0; j < PER; ++j) n += v[j] > -kInf && order_key(v[j]) >= cand;
        if (__reduce_add_sync(FULL, (unsigned)n) >= (unsigned)k) res = cand;
    }
    if (DT == 1 && !(res & 0x80000000u)) res |= 0xffffu;  // a negative value: its key ends in ones
    const float t = from_order_key(res);
    int ng = 0;
#pragma unroll
    for (int j = 0; j < PER; ++j) ng += v[j] > t;
    const int g = (int)__reduce_add_sync(FULL, (unsigned)ng);  // < k
    const int room = kTopMax - g;
    int wg = 0, wt = 0;  // written so far (greater, tied)
#pragma unroll
    for (int j = 0; j < PER; ++j) {
        const bool gt = v[j] > t, eq = v[j] == t;
        const unsigned mg = __ballot_sync(FULL, gt), me = __ballot_sync(FULL, eq);
        const unsigned below = (1u << lane) - 1u;
        if (gt) {
            const int o = wg + __popc(mg & below);
            sv[o] = v[j];
            si[o] = ix[j];
        }
        if (eq) {
            const int o = wt + __popc(me & below);
            if (o < room) {
                sv[g + o] = v[j];
                si[g + o] = ix[j];
            }
        }
        wg += __popc(mg);
        wt += __popc(me);
    }
    __syncwarp();
    if (wt > room) C.dropmax = fmaxf(C.dropmax, t);
    C.n = g + min(wt, room);
    C.thr = fmaxf(C.thr, t);
    return C;
}

// the buffer (n <= 64 entries) as a sorted top list
__device__ __noinline__ TopList cand_to_list(const CandState& C, const float* sv, const int* si, int k) {
    const int lane = threadIdx.x & 31;
    TopList L;
    L.reset();
    float av = lane < C.n ? sv[lane] : -kInf, bv = 32 + lane < C.n ? sv[32 + lane] : -kInf;
    int ai = lane < C.n ? si[lane] : INT_MAX, bi = 32 + lane < C.n ? si[32 + lane] : INT_MAX;
    __syncwarp();
    top_sort(av, ai, lane);
    top_sort(bv, bi, lane);
    top_merge(av, ai, bv, bi, L.av, L.ai, L.bv, L.bi, lane);
    L.dropmax = C.dropmax;
    L.thr = fmaxf(C.thr, L.entry(k - 1));
    return L;
}

// Next bf16 value below x (x a bf16 value, not NaN, not -inf): with it,
// "y >= x" is "y > bf16_pred(x)" for every bf16 y.
__device__ __forceinline__ uint32_t bf16_pred(uint32_t xb) {
    if (xb == 0x0000u || xb == 0x8000u) return 0x8001u;  // +-0 -> the negative denormal next to zero
    return (xb & 0x8000u) ? xb + 1u : xb - 1u;
}

// candidate bits of the 8 tokens of a bf16 vector: bit e iff token e > the
// bf16 pair tt (packed max, then compare with tt; NaN halves lose the max)
__device__ __forceinline__ uint32_t bf16_vec_bits(const uint4& d, uint32_t tt) {
    const uint32_t z0 = bf2_max(d.x, tt) ^ tt, z1 = bf2_max(d.y, tt) ^ tt;
    const uint32_t z2 = bf2_max(d.z, tt) ^ tt, z3 = bf2_max(d.w, tt) ^ tt;
    return (uint32_t)((z0 & 0xffffu) != 0) | ((uint32_t)((z0 >> 16) != 0) << 1) |
           ((uint32_t)((z1 & 0xffffu) != 0) << 2) | ((uint32_t)((z1 >> 16) != 0) << 3) |
           ((uint32_t)((z2 & 0xffffu) != 0) << 4) | ((uint32_t)((z2 >> 16) != 0) << 5) |
           ((uint32_t)((z3 & 0xffffu) != 0) << 6) | ((uint32_t)((z3 >> 16) != 0) << 7);
}

// Append the wanted tokens of this lane's flagged vectors (bit j of vf: the
// vector staged at st[j * 32 + lane]) to the buffer, compacting it when they
// do not fit (then the rest are re-tested against the raised threshold).
// Out of line: the scan keeps no token array in registers across it.
template <int DT>
__device__ __forceinline__ float staged_token(const uint4* st, int j, int e, int lane) {
    const uint4* vp = st + j * 32 + lane;
    if constexpr (DT == 1) return __uint_as_float((uint32_t)reinterpret_cast<const unsigned short*>(vp)[e] << 16);
    else return reinterpret_cast<const float*>(vp)[e];
}

template <int DT>
__device__ __noinline__ CandState cand_append(CandState C, float* sv, int* si, const uint4* st, unsigned vf,
                                              int i0, int k) {
    constexpr int VW = DT == 1 ? 8 : 4;
    const int lane = threadIdx.x & 31;
    __syncwarp();
    while (true) {
        // candidate bits, VW per flagged vector
        uint64_t mask = 0;
        if constexpr (DT == 1) {
            // packed test against the pair tt (a superset: +-0 may tie), then the exact test per bit
            const bool strict = C.thr == -kInf || !(C.dropmax < C.thr);
            const uint32_t tb = __float_as_uint(C.thr) >> 16;
            const uint32_t t1 = strict ? tb : bf16_pred(tb);
            const uint32_t tt = t1 | (t1 << 16);
            for (unsigned m = vf; m; m &= m - 1) {
                const int j = __ffs(m) - 1;
                mask |= (uint64_t)bf16_vec_bits(st[j * 32 + lane], tt) << (j * VW);
            }
            for (uint64_t m = mask; m; m &= m - 1) {
                const int b = __ffsll((long long)m) - 1;
                if (!C.wants(staged_token<DT>(st, b / VW, b % VW, lane))) mask &= ~(1ull << b);
            }
        } else {
            for (unsigned m = vf; m; m &= m - 1) {
                const int j = __ffs(m) - 1;
                uint32_t b = 0;
#pragma unroll
                for (int e = 0; e < 4; ++e) b |= (uint32_t)C.wants(staged_token<DT>(st, j, e, lane)) << e;
                mask |= (uint64_t)b << (j * VW);
            }
        }
        const int cnt = __popcll(mask);
        int off = cnt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(FULL, off, o);
            if (lane >= o) off += t;
        }
        const int total = __shfl_sync(FULL, off, 31);
        off -= cnt;
        const bool fits = C.n + off + cnt <= kCandCap;
        if (fits) {
            int o = C.n + off;
            for (uint64_t m = mask; m; m &= m - 1) {
                const int b = __ffsll((long long)m) - 1, j = b / VW, e = b % VW;
                sv[o] = staged_token<DT>(st, j, e, lane);
                si[o] = i0 + 32 * VW * j + e;
                ++o;
            }
        }
        const unsigned done = __ballot_sync(FULL, fits);  // a prefix of the lanes
        if (done == FULL) {
            C.n += total;
            __syncwarp();
            return C;
        }
        const int last = 31 - __clz(done | 1u);
        C.n += done ? __shfl_sync(FULL, off + cnt, last) : 0;
        if (fits) vf = 0;
        __syncwarp();
        C = cand_compact<DT>(C, sv, si, k);
    }
}

// Flagged vectors wait in a per-warp queue in shared memory (their 16 bytes
// and their index in the row); one iteration adds at most 32 x NV.
constexpr int kTQueueCap = 32 + 32 * PPS_TRUNC_UNITS;

// Work off the queue, one vector per lane, 32 at a time.
template <int DT>
__device__ __noinline__ CandState topk_flush(CandState C, float* sv, int* si, const uint4* qv, const uint32_t* qi,
                                             int qn, int k) {
    constexpr int VW = DT == 1 ? 8 : 4;
    const int lane = threadIdx.x & 31;
    __syncwarp();
    for (int base = 0; base < qn; base += 32) {
        const bool mine = base + lane < qn;
        const int i0 = mine ? (int)(qi[base + lane] * VW) : 0;
        C = cand_append<DT>(C, sv, si, qv + base, mine ? 1u : 0u, i0, k);
    }
    // raise the threshold early: a stale one lets through many more tokens
    if (C.n >= PPS_TRUNC_EAGER) C = cand_compact<DT>(C, sv, si, k);
    return C;
}

// One iteration of the fast scan (NV vectors per lane, d[j] = vector vfirst +
// 32 j): a packed max tree per lane and a vote; vectors with a logit at or
// over the threshold are queued, and the queue is worked off once it holds 32.
template <int DT>
__device__ __forceinline__ void topk_step(CandState& C, float* sv, int* si, uint4* qv, uint32_t* qi, int& qn,
                                          const uint4 (&d)[PPS_TRUNC_UNITS], int64_t vfirst, int k) {
    constexpr int NV = PPS_TRUNC_UNITS;
    const int lane = threadIdx.x & 31;
    unsigned vf = 0;
    if constexpr (DT == 1) {
        const uint32_t tb = __float_as_uint(C.thr) >> 16;  // a bf16 value (or -inf) on bf16 rows
        const uint32_t t2 = tb | (tb << 16);
        uint32_t mv[NV];
#pragma unroll
        for (int j = 0; j < NV; ++j) mv[j] = bf2_max(bf2_max(d[j].x, d[j].y), bf2_max(d[j].z, d[j].w));
        uint32_t m = mv[0];
#pragma unroll
        for (int j = 1; j < NV; ++j) m = bf2_max(m, mv[j]);
        const bool hit = bf2_any_ge(m, t2);
        if (!__any_sync(FULL, hit)) return;
        if (hit) {
#pragma unroll
            for (int j = 0; j < NV; ++j) vf |= (unsigned)bf2_any_ge(mv[j], t2) << j;
        }
    } else {
        float mv[NV];
#pragma unroll
        for (int j = 0; j < NV; ++j) mv[j] = vecs_max<DT>(d, j, 1);
        float m = mv[0];
#pragma unroll
        for (int j = 1; j < NV; ++j) m = fmaxf(m, mv[j]);
        const bool hit = m >= C.thr;
        if (!__any_sync(FULL, hit)) return;
        if (hit) {
#pragma unroll
            for (int j = 0; j < NV; ++j) vf |= (unsigned)(mv[j] >= C.thr) << j;
        }
    }
    const int n = __popc(vf);
    int off = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(FULL, off, o);
        if (lane >= o) off += t;
    }
    const int total = __shfl_sync(FULL, off, 31);
    off += qn - n;
#pragma unroll
    for (int j = 0; j < NV; ++j)
        if ((vf >> j) & 1u) {
            qv[off] = d[j];
            qi[off] = (uint32_t)(vfirst + 32 * j);
            ++off;
        }
    qn += total;
    if (qn >= 32) {
        C = topk_flush<DT>(C, sv, si, qv, qi, qn, k);
        qn = 0;
    }
}

// The fast scan of the full vectors [v0, vend) of a row: iterations of NV
// vectors 32 apart per lane; in the last, partial one the vectors past vend
// read as -inf.  The first iteration also seeds the threshold.
template <int DT>
__device__ __forceinline__ void topk_scan(CandState& C, float* sv, int* si, uint4* qv, uint32_t* qi,
                                          const char* row, int64_t v0, int64_t vend, int k) {
    constexpr int NV = PPS_TRUNC_UNITS;
    constexpr int STEP = 32 * NV;
    const int lane = threadIdx.x & 31;
    const uint32_t ninf = DT == 1 ? 0xff80ff80u : 0xff800000u;
    const uint4 fill = make_uint4(ninf, ninf, ninf, ninf);
    const int64_t n_it = (vend - v0 + STEP - 1) / STEP;
    const uint4* p = reinterpret_cast<const uint4*>(row) + v0 + lane;
    int qn = 0;
    for (int64_t it = 0; it < n_it; ++it) {
        const int64_t vb = v0 + it * STEP + lane;
        uint4 d[NV];
        if (v0 + (it + 1) * STEP <= vend) {
#pragma unroll
            for (int j = 0; j < NV; ++j) d[j] = ldg_stream(p + 32 * j);
        } else {
#pragma unroll
            for (int j = 0; j < NV; ++j) d[j] = vb + 32 * j < vend ? ldg_stream(p + 32 * j) : fill;
        }
        p += STEP;
        if (it == 0) C.thr = seed_thr<DT>(d, k);
        topk_step<DT>(C, sv, si, qv, qi, qn, d, vb, k);
    }
    if (qn > 0) C = topk_flush<DT>(C, sv, si, qv, qi, qn, k);
}

// Scalar-load path: the last partial iteration of a segment, the ragged
// vector of a row and unaligned rows, one vector per lane at a time.
template <int DT>
__device__ __noinline__ TopList topk_tail(TopList L, const char* row, int64_t V, int64_t base, int64_t v1, int k) {
    constexpr int VW = DT == 1 ? 8 : 4;
    const int lane = threadIdx.x & 31;
    for (; base < v1; base += 32) {
        const int64_t v = base + lane;
        float cv[VW];
        int ci[VW];
        uint4 d = make_uint4(0, 0, 0, 0);
        int64_t nt = 0;
        if (v < v1) {
            d = load_scalar<DT>(row, v, V);
            nt = min((int64_t)VW, V - v * VW);
        }
#pragma unroll
        for (int e = 0; e < VW; ++e) {
            const float x = vec_token<DT>(d, e);
            cv[e] = (e < nt && x == x) ? x : -kInf;
            ci[e] = (int)(v * VW + e);
        }
        top_offer<VW>(L, cv, ci, k, lane);
    }
    return L;
}

template <int DT, bool VEC>
__device__ __forceinline__ void topk_segment(TopList& L, const char* row, int64_t V, int64_t v0, int64_t v1, int k,
                                             float* sv, int* si, uint4* qv, uint32_t* qi) {
    constexpr int VW = DT == 1 ? 8 : 4;
    const int64_t nfull = V / VW;
    const int64_t vend = VEC ? min(v1, nfull) : v0;
    if (vend > v0) {
        CandState C{-kInf, -kInf, 0};
        topk_scan<DT>(C, sv, si, qv, qi, row, v0, vend, k);
        if (C.n > kTopMax) C = cand_compact<DT>(C, sv, si, k);
        L = cand_to_list(C, sv, si, k);
    }
    // the row's ragged last vector, or a whole unaligned segment
    if (vend < v1) L = topk_tail<DT>(L, row, V, vend > v0 ? vend : v0, v1, k);
}

// ---------------------------------------------------------------- finishing a truncated row

template <int DT>
__device__ __noinline__ int64_t count_logit(const char* row, int64_t V, float x) {
    const int lane = threadIdx.x & 31;
    long long n = 0;
    for (int64_t i = lane; i < V; i += 32) n += load_logit<DT>(row, i) == x;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(FULL, n, o);
    return (int64_t)n;
}

// Top-p on the kept-by-top-k set: the list's entries with logit >= lk (a
// prefix, in top order) plus `extra` more tokens of logit lk that the list
// could not hold.  Lane 0 walks them in ascending order, exactly as the
// definition sums; returns the smallest kept logit (every token >= it stays).
__device__ __noinline__ float top_p_keep(const TopList& L, float lk, int64_t extra, float top_p, float T,
                                         float* s_val) {
    const int lane = threadIdx.x & 31;
    s_val[lane] = L.av;
    s_val[32 + lane] = L.bv;
    __syncwarp();
    float keep = lk;
    if (lane == 0) {
        int nk = 0;
        while (nk < kTopMax && s_val[nk] > -kInf && s_val[nk] >= lk) ++nk;
        const double top = (double)s_val[0], Td = (double)T, cut = 1.0 - (double)top_p;
        const double ex = exp(((double)lk - top) / Td);
        double Z = 0.0;
        for (int64_t t = 0; t < extra; ++t) Z += ex;
        for (int j = nk - 1; j >= 0; --j) Z += exp(((double)s_val[j] - top) / Td);
        double run = 0.0;
        for (int64_t t = 0; t < extra; ++t) run += ex / Z;
        float kv = s_val[0];
        for (int j = nk - 1; j >= 0; --j) {
            run += exp(((double)s_val[j] - top) / Td) / Z;
            if (j > 0 && s_val[j - 1] == s_val[j]) continue;  // not the end of its group
            if ((double)s_val[j] == top) break;               // the top group stays
            if (run <= cut) {
                kv = s_val[j - 1];
            } else {
                kv = s_val[j];
                break;
            }
        }
        keep = kv;
    }
    __syncwarp();
    return __shfl_sync(FULL, keep, 0);
}

// lower 32 of two lists sorted ascending by (key, token): into x
__device__ __forceinline__ void merge_low_f(float& xk, int& xi, float yk, int yi, int lane) {
    const float rk = __shfl_sync(FULL, yk, 31 - lane);
    const int ri = __shfl_sync(FULL, yi, 31 - lane);
    if (lex_less(rk, ri, xk, xi)) {
        xk = rk;
        xi = ri;
    }
#pragma unroll
    for (int stride = 16; stride > 0; stride >>= 1) {
        const float ok = __shfl_xor_sync(FULL, xk, stride);
        const int oi = __shfl_xor_sync(FULL, xi, stride);
        const bool lower = (lane & stride) == 0;
        const bool o_less = lex_less(ok, oi, xk, xi);
        if (lower ? o_less : (!o_less && !(ok == xk && oi == xi))) {
            xk = ok;
            xi = oi;
        }
    }
}
template <int DT, bool VERIFY, bool BLK>
__device__ __noinline__ void finalize_trunc(const RaceArgs& a, int64_t r, const TopList& L, int kr, int kp,
                                            float* s_val, Blk bk, uint32_t* scratch) {
    const int lane = threadIdx.x & 31;
    const int k = a.top_k;
    const float lk = L.entry(k - 1);  // l_(k); -inf when the row has fewer than k usable tokens
    const bool over = lk > -kInf && L.dropmax >= lk;
    const char* row = reinterpret_cast<const char*>(a.logits) + (size_t)r * (size_t)a.stride * (DT == 1 ? 2 : 4);
    const uint64_t key = a.key[r], ctx = a.ctx[r];
    const uint32_t pos = a.pos[r];
    float keep = lk;
    if (a.top_p < 1.0f) {
        int64_t extra = 0;
        if (over) {
            const int in_list = __popc(__ballot_sync(FULL, L.av == lk)) + __popc(__ballot_sync(FULL, L.bv == lk));
            extra = count_logit<DT>(row, a.V, lk) - in_list;
        }
        keep = top_p_keep(L, lk, extra, a.top_p, a.T, s_val);
    }
    if (over && keep <= lk) {
        // the tie group of l_(k) stays but is not all in the list: exact race
        // over every token with logit >= l_(k), one pass of the scalar path
        WarpList W;
        W.reset(kp, kr);
        SlowState st{W};
        st = tail_loop<DT, BLK>(st, row, a.V, 0, a.nv, a.c, key, ctx, pos, lk, bk);
        finalize_row<DT, VERIFY, BLK>(a, r, st.L.lk, st.L.li, st.L.drop(), kr, kp, lane, bk, scratch);
        return;
    }
    // S = the list's entries with logit >= keep: the race's fp32 keys, the 32
    // smallest in lane order; finalize_row re-keys near ties in fp64 (S is
    // complete, so nothing was dropped: drop bound +inf)
    float ka = kInf, kb = kInf;
    int ia = L.ai, ib = L.bi;
    // proposal rows of the augmented race: the tokens' block arrivals
    auto list_key = [&](int i, float l) {
        const uint32_t w = word_of(key, ctx, pos, i, 1);
        if constexpr (BLK) return block_key_of(key, ctx, pos, i, w, l, a.c, bk.b, bk.B, bk.invB());
        return key32(w, l, a.c);
    };
    if (L.av > -kInf && L.av >= keep) ka = list_key(ia, L.av);
    if (L.bv > -kInf && L.bv >= keep) kb = list_key(ib, L.bv);
    if (ka == kInf) ia = INT_MAX;
    if (kb == kInf) ib = INT_MAX;
    warp_sort(ka, ia, lane);
    warp_sort(kb, ib, lane);
    merge_low_f(ka, ia, kb, ib, lane);
    finalize_row<DT, VERIFY, BLK>(a, r, ka, ia, kInf, kr, kp, lane, bk);
}

template <int DT, bool VERIFY, bool BLK>
__device__ __noinline__ void finish_trunc_segment(const RaceArgs& a, int64_t r, int64_t gw, int64_t NW, int64_t v0,
                                                  int64_t v1, TopList L, int kr, int kp, float* s_val, Blk bk,
                                                  uint32_t* scratch) {
    const int lane = threadIdx.x & 31;
    const int64_t nv = a.nv;
    bool final_here = v0 == 0 && v1 == nv;
    if (!final_here) {
        // publish this segment's list; the last warp of the row merges all segments
        TruncPartial* P = a.tpartials + (gw + r);
        P->v[lane] = L.av;
        P->v[32 + lane] = L.bv;
        P->idx[lane] = L.ai;
        P->idx[32 + lane] = L.bi;
        if (lane == 0) P->dropmax = L.dropmax;
        __threadfence();
        __syncwarp();
        const int64_t first_w = warp_of(r * nv, a.total, NW);
        const int64_t last_w = warp_of(r * nv + nv - 1, a.total, NW);
        unsigned last = 0;
        if (lane == 0) {
            unsigned t = atomicAdd(a.row_cnt + r, 1u);
            last = t == (unsigned)(last_w - first_w);
            if (last) a.row_cnt[r] = 0u;
        }
        final_here = __shfl_sync(FULL, last, 0) != 0;
        if (final_here) {
            __threadfence();
            L.reset();
            for (int64_t ww = first_w; ww <= last_w; ++ww) {
                const TruncPartial* Q = a.tpartials + (ww + r);
                L.insert_sorted(__ldcg(Q->v + lane), __ldcg(Q->idx + lane), a.top_k, lane);
                L.insert_sorted(__ldcg(Q->v + 32 + lane), __ldcg(Q->idx + 32 + lane), a.top_k, lane);
                L.dropmax = fmaxf(L.dropmax, __ldcg(&Q->dropmax));
            }
        }
    }
    if (final_here) {
        finalize_trunc<DT, VERIFY, BLK>(a, r, L, kr, kp, s_val, bk, scratch);
        if constexpr (VERIFY) sequence_ticket(a, r, lane);
    }
}

// ---------------------------------------------------------------- the kernel

template <int DT, bool VERIFY, bool VEC, bool BLK>
__global__ void __launch_bounds__(kThreads, PPS_TRUNC_MIN_BLOCKS) trunc_kernel(const RaceArgs a) {
    __shared__ float s_val[kTopMax];
    __shared__ float s_cv[kCandCap];
    __shared__ int s_ci[kCandCap];
    __shared__ uint4 s_qv[kTQueueCap];
    __shared__ uint32_t s_qi[kTQueueCap];
    pdl_wait();  // the previous kernel's outputs and the workspace it used
    pdl_launch_dependents();
    const int64_t NW = a.G;
    const int64_t gw = blockIdx.x;
    const int64_t g0 = gw * a.total / NW, g1 = (gw + 1) * a.total / NW;
    const int64_t nv = a.nv;
    const size_t esz = DT == 1 ? 2 : 4;

    for (int64_t r = g0 / nv; g0 < g1 && r < a.n_rows && r * nv < g1; ++r) {
        const int64_t v0 = max(g0, r * nv) - r * nv, v1 = min(g1, (r + 1) * nv) - r * nv;
        int kr = 1;
        if (!VERIFY) {
            kr = a.row_k ? __ldg(a.row_k + r) : a.K;
            kr = max(1, min(kr, a.K));
        }
        const int kp = min(32, 2 * kr + 1);
        const char* row = reinterpret_cast<const char*>(a.logits) + (size_t)r * (size_t)a.stride * esz;
        TopList L;
        L.reset();
        topk_segment<DT, VEC>(L, row, a.V, v0, v1, a.top_k, s_cv, s_ci, s_qv, s_qi);
        Blk bk;
        if constexpr (BLK) {
            bk.b = __ldg(a.row_block + r);
            bk.B = a.n_blocks;
        }
        finish_trunc_segment<DT, VERIFY, BLK>(a, r, gw, NW, v0, v1, L, kr, kp, s_val, bk,
                                              reinterpret_cast<uint32_t*>(s_ci));
    }
}
