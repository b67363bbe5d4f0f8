// pps_lmhead.cuh -- the keyed race fused into the LM-head GEMM (sm_103a).
// Included by pps_race.cu, whose list finishing, near-tie re-keying, IID
// epilogue and tree walk it reuses (one translation unit).
//
// logits[r, i] = sum_j hidden[r, j] W[i, j]   (bf16 operands, fp32 accumulate)
//
// is the last layer of the target (or draft) model.  The batched-target
// algorithm evaluates the target once for every context of a draft block
// (App. B, the cost remark after the direct finite-support MPFR algorithm);
// here the race of Alg. 2 runs on each accumulator tile while it sits in
// tensor memory, so no logits row is ever written to HBM.
//
// GEMM.  One CTA per SM, warp-specialised: warp 0 issues TMA loads of
// 128 x 64 hidden tiles and 256 x 64 weight tiles (128-byte swizzle) into a
// 4-stage shared-memory ring; one thread of warp 1 issues tcgen05.mma
// (M = 128, N = 256, K = 16, bf16 -> fp32) into one of two 256-column
// accumulators in tensor memory; warps 2..9 read the finished accumulator
// with tcgen05.ld (thread = one row, 128 columns each) while the next tile
// accumulates in the other.  CTA c owns row block c % MB and the c / MB-th
// slice of the vocabulary, so the MB CTAs of a slice read the same weight
// tiles at the same time (they stay in L2) and a thread's row stays the same
// over its whole slice.
//
// Race epilogue.  Each thread keeps, for its row and slice half, the kp
// smallest fp32 race keys (key32, a monotone image of s = ln E - l/T) with
// their tokens and logits, and a drop bound, exactly like the warp lists of
// the streaming kernel: the same conservative filter (one ex2 per 4 tokens
// when the block's largest word and logit fail it), the same key, the same
// bound update.  A second kernel merges the 2S partial lists of a row and
// finishes it with the streaming kernel's finishing code (completeness test,
// fp64 re-keying of near ties, IID epilogue), taking the logits of the listed
// tokens from the lists; verify rows then walk their sequence.  The result
// is the race of the fp32 accumulators, the same logits that the unfused path
// (pps_lmhead_logits, the same MMA schedule, then the streaming race) reads.
//
// Every wait on an mbarrier gives up after kLmWaitLimit polls: the CTA then
// raises PPS_FLAG_TIMEOUT in the status word, stops issuing work, waits (again
// bounded) for its own copies in flight, frees its tensor memory and returns.
// (<cuda.h>, for CUtensorMap, is included at the top of pps_race.cu.)

namespace lm {

constexpr int BM = 128;                                // rows per tile (TMEM lanes)
constexpr int BN = 256;                                // vocabulary columns per tile
constexpr int BK = 64;                                 // reduction step: 64 bf16 = one 128-byte swizzle row
constexpr int kStages = 4;
constexpr int kEpiWarps = 8;
constexpr int kLmThreads = 32 * (2 + kEpiWarps);       // TMA warp, MMA warp, 8 epilogue warps
constexpr int kStageA = BM * BK * 2;                   // 16 KB
constexpr int kStageB = BN * BK * 2;                   // 32 KB
constexpr int kStageBytes = kStageA + kStageB;
constexpr int kTmemCols = 2 * BN;                      // two fp32 accumulators
constexpr int kMaxSlices = 16;                         // 2 x slices partial lists per row (<= 32)
constexpr int kLmSmem = kStages * kStageBytes + 1024 /* alignment */ + 256 /* barriers, flags */;
constexpr uint32_t kLmWaitLimit = 1u << 22;

// instruction descriptor of tcgen05.mma kind::f16: fp32 accumulator (bits 4-5),
// bf16 A and B (7-9, 10-12), both K-major (15, 16 = 0), N >> 3 (17-22), M >> 4 (24-28)
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

// ---------------------------------------------------------------- mbarriers
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// Wait for the phase of parity `parity` to complete; false when the CTA is
// aborting or the wait gave up (which starts the abort).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort) {
    for (uint32_t n = 0; n < kLmWaitLimit; ++n) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort) return false;
    }
    *abort = 1;
    return false;
}

// ---------------------------------------------------------------- TMA
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, uint32_t bar, int x, int y) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(x), "r"(y)
        : "memory");
}
__device__ __forceinline__ void tma_prefetch_map(const CUtensorMap* map) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ---------------------------------------------------------------- tensor memory and tcgen05
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
// arrive on `bar` once every tcgen05.mma issued so far by this thread has completed
__device__ __forceinline__ void tc_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
// D (tmem) = A (smem) x B (smem)^T [+ D]
__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(kIdesc), "r"(accumulate)
        : "memory");
}
// thread t of the warp reads lane (taddr lane + t), 32 consecutive 32-bit columns
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
          "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]),
          "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
          "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr)
        : "memory");
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// Shared-memory matrix descriptor of a K-major tile written by TMA with the
// 128-byte swizzle: rows of 128 bytes, 8-row groups 1024 bytes apart (stride
// byte offset), start address >> 4 in bits 0-13, descriptor version 1 in bits
// 46-47, swizzle mode 2 (128 B) in bits 61-63.  The leading byte offset is
// not used by swizzled K-major layouts.  Tiles start on 1024-byte boundaries
// (base offset 0); the k-th 16-element step of a 64-element row is the
// start address + 32 k bytes.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)(1024 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

}  // namespace lm

namespace lm {

// one partial list of the race epilogue: a thread's row over one slice half
constexpr int kLmKP = 10;  // longest kept list: K <= 8 drafts, kp = K + 2
struct alignas(16) LmPartial {
    float key[kLmKP];    // fp32 race keys (key32), ascending with (key, token)
    int32_t idx[kLmKP];  // tokens (INT_MAX: empty)
    float logit[kLmKP];  // the tokens' fp32 logits (the accumulator values)
    float theta;         // every token of the range left out has key32 >= theta
    int32_t pad;
};
static_assert(sizeof(LmPartial) == 128, "one 128-byte partial list");

struct LmArgs {
    int64_t n_rows, V, d;
    int MB;  // row blocks of BM rows
    int S;   // vocabulary slices per row block
    int NT;  // vocabulary tiles of BN columns
    int KB;  // reduction steps of BK
    // store epilogue: logits [n_rows, ldo] fp32
    float* out;
    int64_t ldo;
    // race epilogue
    const uint64_t* key;
    const uint64_t* ctx;
    const uint32_t* pos;
    const int32_t* row_k;  // nullable (K for every row)
    int K;                 // list length (1: target race)
    float c;               // log2(e) / T
    LmPartial* partials;   // [n_rows][2 S]
    uint32_t* status;
};

// Store epilogue: the thread's 32 accumulator values of its row go to the logits matrix.
struct StoreEpi {
    float* p = nullptr;  // the row's output, nullptr for rows past the end
    int64_t V = 0;
    __device__ __forceinline__ void init(const LmArgs& a, int64_t row, int, int) {
        V = a.V;
        p = row < a.n_rows ? a.out + row * a.ldo : nullptr;
    }
    __device__ __forceinline__ void chunk(const uint32_t (&v)[32], int64_t n) {
        if (p == nullptr) return;
        float* q = p + n;
        if (n + 32 <= V && (reinterpret_cast<uintptr_t>(q) & 15u) == 0) {
#pragma unroll
            for (int j = 0; j < 32; j += 4)
                *reinterpret_cast<float4*>(q + j) = make_float4(__uint_as_float(v[j]), __uint_as_float(v[j + 1]),
                                                                __uint_as_float(v[j + 2]), __uint_as_float(v[j + 3]));
        } else {
#pragma unroll
            for (int j = 0; j < 32; ++j)
                if (n + j < V) q[j] = __uint_as_float(v[j]);
        }
    }
    __device__ __forceinline__ void finish(const LmArgs&, int64_t, int, int) {}
};

// Race epilogue: the kp smallest (key32, token) of the thread's row over its
// slice half, kept sorted in registers (kp = min(KP, k + 2): the k the row
// needs, one spare for near-tie re-keying at the boundary and one whose key
// bounds what was left out), and the filter bound tf, lowered like the
// streaming kernel's warp lists: to entry kp-1 (nothing at or above it can
// enter) and to filter_slack of entry k-1 (nothing above it can tie with the
// row's k-th key).  Every token left out has key32 >= min(entry kp-1, tf).
template <int KP>
struct RaceEpi {
    RowPhilox rp;
    bool live = false;
    int64_t V = 0;
    float c = 0.f, tf = 0.f, tz = 0.f;
    int kr = 1, kp = 1;
    float k[KP], l[KP];
    int i[KP];

    __device__ __forceinline__ float entry_key(int m) const {
        float t = kInf;
#pragma unroll
        for (int e = 0; e < KP; ++e)
            if (e == m) t = k[e];
        return t;
    }
    __device__ __forceinline__ int entry_idx(int m) const {
        int t = INT_MAX;
#pragma unroll
        for (int e = 0; e < KP; ++e)
            if (e == m) t = i[e];
        return t;
    }
    __device__ __forceinline__ void init(const LmArgs& a, int64_t row, int, int) {
        live = row < a.n_rows;
        V = a.V;
        c = a.c;
        kr = 1;
        if (live && a.row_k) kr = __ldg(a.row_k + row);
        else kr = a.K;
        kr = max(1, min(kr, a.K));
        kp = min(KP, kr + 2);
#pragma unroll
        for (int e = 0; e < KP; ++e) {
            k[e] = kInf;
            l[e] = 0.f;
            i[e] = INT_MAX;
        }
        tf = kInf;
        tz = filter_tz(kInf);
        if (live) rp.init_thread(__ldg(a.key + row), __ldg(a.ctx + row), __ldg(a.pos + row));
    }
    // insert (ck, ci, cl) if it is below entry kp-1, then lower the bound
    __device__ __forceinline__ void offer(float ck, int ci, float cl) {
        if (!lex_less(ck, ci, entry_key(kp - 1), entry_idx(kp - 1))) return;
        bool placed = false;
#pragma unroll
        for (int m = KP - 1; m >= 0; --m) {
            if (!placed) {
                if (m > 0 && lex_less(ck, ci, k[m - 1], i[m - 1])) {
                    k[m] = k[m - 1];
                    i[m] = i[m - 1];
                    l[m] = l[m - 1];
                } else {
                    k[m] = ck;
                    i[m] = ci;
                    l[m] = cl;
                    placed = true;
                }
            }
        }
        tf = fminf(tf, fminf(entry_key(kp - 1), filter_slack(entry_key(kr - 1))));
        tz = filter_tz(tf);
    }
    // The 32 tokens n..n+31 of the thread's row: the unrolled scan only sets a bit per token
    // over the filter cut; the rare survivors are keyed and offered afterwards, one at a time
    // (their words recomputed), so the insertion code appears once, outside the scan.
    __device__ __forceinline__ void chunk(const uint32_t (&v)[32], int64_t n) {
        if (!live) return;
        uint32_t pass = 0;
#pragma unroll
        for (int b = 0; b < 8; ++b) {
            const int64_t t0 = n + 4 * b;
            if (t0 < V) {
                const uint4 w = rp.block((uint32_t)(t0 >> 2));
                const uint32_t wq[4] = {w.x, w.y, w.z, w.w};
                const float lq[4] = {__uint_as_float(v[4 * b]), __uint_as_float(v[4 * b + 1]),
                                     __uint_as_float(v[4 * b + 2]), __uint_as_float(v[4 * b + 3])};
                // the block's largest word with its largest logit passes whenever one of its tokens would
                const uint32_t wm = max(max(wq[0], wq[1]), max(wq[2], wq[3]));
                const float lm = fmaxf(fmaxf(lq[0], lq[1]), fmaxf(lq[2], lq[3]));
                if (filter_pass(wm, lm, c, tz)) {
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        if (t0 + e < V && filter_pass(wq[e], lq[e], c, tz)) pass |= 1u << (4 * b + e);
                }
            }
        }
#pragma unroll 1
        while (pass) {
            const int j = __ffs(pass) - 1;
            pass &= pass - 1;
            const int64_t tok = n + j;
            const uint4 w = rp.block((uint32_t)(tok >> 2));
            const uint32_t wj = (j & 3) == 0 ? w.x : (j & 3) == 1 ? w.y : (j & 3) == 2 ? w.z : w.w;
            float lj = 0.f;
#pragma unroll
            for (int e = 0; e < 32; ++e)
                if (e == j) lj = __uint_as_float(v[e]);
            // the bound may have dropped since the scan: test again against the current one
            if (filter_pass(wj, lj, c, tz)) offer(key32(wj, lj, c), (int)tok, lj);
        }
    }
    __device__ __forceinline__ void finish(const LmArgs& a, int64_t row, int slice, int half) {
        if (!live) return;
        LmPartial* P = a.partials + (row * (2 * a.S) + 2 * slice + half);
#pragma unroll
        for (int e = 0; e < kLmKP; ++e) {
            const bool use = e < KP && e < kp;
            P->key[e] = use ? k[e < KP ? e : 0] : kInf;
            P->idx[e] = use ? i[e < KP ? e : 0] : INT_MAX;
            P->logit[e] = use ? l[e < KP ? e : 0] : 0.f;
        }
        P->theta = fminf(entry_key(kp - 1), tf);
    }
};

}  // namespace lm

namespace lm {

// Shared memory: kStages x (A tile 16 KB | B tile 32 KB), 1024-byte aligned,
// then the mbarriers full[s], empty[s], tfull[2], tempty[2], the abort flag
// and the tensor-memory address written by tcgen05.alloc.
template <class Epi>
__global__ void __launch_bounds__(kLmThreads, 1)
    lmhead_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, const LmArgs a) {
    extern __shared__ uint8_t lm_smem_raw[];
    const uint32_t raw = smem_u32(lm_smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* gbase = lm_smem_raw + (base - raw);
    const uint32_t bars = base + kStages * kStageBytes;
    auto full = [&](uint32_t s) { return bars + 8u * s; };
    auto empty = [&](uint32_t s) { return bars + 8u * (kStages + s); };
    auto tfull = [&](uint32_t x) { return bars + 8u * (2 * kStages + x); };
    auto tempty = [&](uint32_t x) { return bars + 8u * (2 * kStages + 2 + x); };
    volatile int* abort = reinterpret_cast<volatile int*>(gbase + kStages * kStageBytes + 8 * (2 * kStages + 4));
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + kStages * kStageBytes + 8 * (2 * kStages + 4) + 16);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int mb = (int)(blockIdx.x % (unsigned)a.MB), slice = (int)(blockIdx.x / (unsigned)a.MB);
    const int t0 = (int)((int64_t)slice * a.NT / a.S), t1 = (int)((int64_t)(slice + 1) * a.NT / a.S);
    const int m0 = mb * BM;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(full(s), 1);
            mbar_init(empty(s), 1);
        }
        for (int x = 0; x < 2; ++x) {
            mbar_init(tfull(x), 1);
            mbar_init(tempty(x), kEpiWarps);
        }
        *abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_map(&tmA);
        tma_prefetch_map(&tmB);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        // ---- TMA producer
        if (lane == 0) {
            uint32_t it = 0;
            for (int t = t0; t < t1 && !*abort; ++t) {
                const int n0 = t * BN;
                for (int kb = 0; kb < a.KB; ++kb) {
                    const uint32_t s = it % kStages, ph = (it / kStages) & 1u;
                    if (!mbar_wait(empty(s), ph ^ 1u, abort)) break;
                    const uint32_t sa = base + s * kStageBytes;
                    mbar_expect_tx(full(s), kStageBytes);
                    tma_load_2d(sa, &tmA, full(s), kb * BK, m0);
                    tma_load_2d(sa + kStageA, &tmB, full(s), kb * BK, n0);
                    ++it;
                }
            }
            // the copies of the last stages may still be landing if the MMA warp gave up:
            // wait (bounded) for each of them before the CTA leaves
            const uint32_t from = it > (uint32_t)kStages ? it - kStages : 0u;
            for (uint32_t j = from; j < it && *abort; ++j)
                for (uint32_t n = 0; n < kLmWaitLimit && !mbar_try_wait(full(j % kStages), (j / kStages) & 1u); ++n) {
                }
        }
    } else if (warp == 1) {
        // ---- MMA issuer (one thread)
        if (lane == 0) {
            uint32_t it = 0, tc = 0;
            for (int t = t0; t < t1 && !*abort; ++t, ++tc) {
                const uint32_t acc = tc & 1u, aph = (tc >> 1) & 1u;
                if (!mbar_wait(tempty(acc), aph ^ 1u, abort)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + acc * BN;
                bool ok = true;
                for (int kb = 0; kb < a.KB; ++kb) {
                    const uint32_t s = it % kStages, ph = (it / kStages) & 1u;
                    if (!mbar_wait(full(s), ph, abort)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t da = sw128_desc(base + s * kStageBytes);
                    const uint64_t db = sw128_desc(base + s * kStageBytes + kStageA);
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k)
                        tc_mma(d_tmem, da + 2u * (uint32_t)k, db + 2u * (uint32_t)k, (kb | k) != 0 ? 1u : 0u);
                    tc_commit(empty(s));  // frees the stage once these MMAs have read it
                    ++it;
                }
                if (!ok) break;
                tc_commit(tfull(acc));  // the tile's accumulator is complete
            }
        }
    } else {
        // ---- epilogue: thread = row m0 + 32 q + lane, columns [128 half, 128 half + 128) of each tile
        const int q = warp & 3, half = (warp - 2) >> 2;
        const int64_t row = (int64_t)m0 + 32 * q + lane;
        Epi epi;
        epi.init(a, row, slice, half);
        uint32_t tc = 0;
        for (int t = t0; t < t1; ++t, ++tc) {
            const uint32_t acc = tc & 1u, aph = (tc >> 1) & 1u;
            int ok = 1;
            if (lane == 0) ok = mbar_wait(tfull(acc), aph, abort) ? 1 : 0;
            if (!__shfl_sync(0xffffffffu, ok, 0)) break;
            tc_fence_after();
            const int64_t n0 = (int64_t)t * BN;
#pragma unroll 1
            for (int ch = 0; ch < 4; ++ch) {
                const uint32_t col = (uint32_t)(half * 128 + ch * 32);
                uint32_t v[32];
                tmem_ld32(tmem + acc * BN + ((uint32_t)(32 * q) << 16) + col, v);
                tmem_wait_ld();
                if (ch == 3) {
                    // the accumulator is in registers: hand it back to the MMA warp
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(tempty(acc));
                }
                epi.chunk(v, n0 + col);
                __syncwarp();
            }
        }
        epi.finish(a, row, slice, half);
    }
    __syncwarp();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
    if (threadIdx.x == 0 && *abort && a.status) atomicOr(a.status, PPS_FLAG_TIMEOUT);
}

}  // namespace lm

namespace lm {

// Logits of a row's listed tokens, from the merged list (<= 32 entries).
struct ListLogits {
    static constexpr bool kDense = false;
    const int* tok;
    const float* val;
    __device__ __forceinline__ float operator()(int64_t i) const {
        float r = 0.f;
#pragma unroll 8
        for (int m = 0; m < 32; ++m)
            if (tok[m] == (int)i) r = val[m];
        return r;
    }
};

// One warp per row: the row's P = 2 S partial lists are staged in shared
// memory (list j in column j), merged by kp rounds of one warp argmin over the
// list heads (as merge_rounds does for the streaming kernel), and the row is
// finished by the streaming kernel's finishing code with the listed logits.
template <bool VERIFY>
__global__ void __launch_bounds__(128) lmhead_finish_kernel(const RaceArgs a, const LmPartial* parts, int P) {
    __shared__ float s_k[4][kLmKP * 32];
    __shared__ int s_i[4][kLmKP * 32];
    __shared__ float s_l[4][kLmKP * 32];
    __shared__ int s_tok[4][32];
    __shared__ float s_val[4][32];
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t r = (int64_t)blockIdx.x * 4 + w;
    if (r >= a.n_rows) return;  // warp-uniform
    int kr = 1;
    if (!VERIFY) {
        kr = a.row_k ? __ldg(a.row_k + r) : a.K;
        kr = max(1, min(kr, a.K));
    }
    const int kp = min(kLmKP, kr + 2);
    float th = kInf;
    if (lane < P) {
        const LmPartial* Q = parts + (r * P + lane);
        th = __ldcg(&Q->theta);
        for (int e = 0; e < kp; ++e) {
            s_k[w][e * 32 + lane] = __ldcg(Q->key + e);
            s_i[w][e * 32 + lane] = __ldcg(Q->idx + e);
            s_l[w][e * 32 + lane] = __ldcg(Q->logit + e);
        }
    }
    __syncwarp();
    int h = 0;
    float hk = lane < P ? s_k[w][lane] : kInf;
    int hi = lane < P ? s_i[w][lane] : INT_MAX;
    float hl = lane < P ? s_l[w][lane] : 0.f;
    float lk = kInf, ll = 0.f;
    int li = INT_MAX;
    for (int m = 0; m < kp; ++m) {
        float bk = hk, bl = hl;
        int bi = hi;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ok = __shfl_xor_sync(FULL, bk, o);
            const int oi = __shfl_xor_sync(FULL, bi, o);
            const float ol = __shfl_xor_sync(FULL, bl, o);
            if (lex_less(ok, oi, bk, bi)) {
                bk = ok;
                bi = oi;
                bl = ol;
            }
        }
        if (bi == INT_MAX) break;
        if (lane == m) {
            lk = bk;
            li = bi;
            ll = bl;
        }
        if (hi == bi) {
            ++h;
            hk = h < kp ? s_k[w][h * 32 + lane] : kInf;
            hi = h < kp ? s_i[w][h * 32 + lane] : INT_MAX;
            hl = h < kp ? s_l[w][h * 32 + lane] : 0.f;
        }
    }
    float d = fminf(hk, th);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) d = fminf(d, __shfl_xor_sync(FULL, d, o));
    s_tok[w][lane] = li;
    s_val[w][lane] = ll;
    __syncwarp();
    finalize_row_lp<0, VERIFY, false>(a, r, lk, li, d, kr, kp, lane, ListLogits{s_tok[w], s_val[w]}, Blk{}, nullptr);
    if constexpr (VERIFY) sequence_ticket(a, r, lane);
}

// ---------------------------------------------------------------- host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
    static std::atomic<EncodeTiledFn> cached{nullptr};
    EncodeTiledFn f = cached.load(std::memory_order_relaxed);
    if (f == nullptr) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess || p == nullptr)
            return nullptr;
        f = reinterpret_cast<EncodeTiledFn>(p);
        cached.store(f, std::memory_order_relaxed);
    }
    return f;
}

// bf16 matrix [rows, cols] with row stride ld elements, loaded as boxes of box_rows x BK (128-byte swizzle)
static bool make_map(CUtensorMap* m, const void* ptr, int64_t rows, int64_t cols, int64_t ld, int box_rows) {
    EncodeTiledFn f = encode_fn();
    if (f == nullptr) return false;
    const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    const cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
    const cuuint32_t es[2] = {1, 1};
    return f(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <class Epi>
static cudaError_t launch_gemm(const CUtensorMap& tA, const CUtensorMap& tB, const LmArgs& a, cudaStream_t st) {
    cudaError_t e = cudaFuncSetAttribute(lmhead_kernel<Epi>, cudaFuncAttributeMaxDynamicSharedMemorySize, kLmSmem);
    if (e != cudaSuccess) return e;
    lmhead_kernel<Epi><<<a.MB * a.S, kLmThreads, kLmSmem, st>>>(tA, tB, a);
    return cudaGetLastError();
}

// the schedule: MB row blocks x S vocabulary slices, S = SMs / MB (1..kMaxSlices, <= NT)
static void schedule(LmArgs& a) {
    a.MB = (int)((a.n_rows + BM - 1) / BM);
    a.NT = (int)((a.V + BN - 1) / BN);
    a.KB = (int)((a.d + BK - 1) / BK);
    int S = device_sm_count() / max(1, a.MB);
    S = max(1, min(S, kMaxSlices));
    a.S = min(S, a.NT);
}

}  // namespace lm

size_t lmhead_workspace_bytes(int64_t n_rows, int32_t n_seq) {
    auto al = [](size_t x) { return (x + 255) & ~(size_t)255; };
    return al(sizeof(lm::LmPartial) * 2 * lm::kMaxSlices * (size_t)n_rows) + al(sizeof(uint32_t) * (size_t)(n_seq > 0 ? n_seq : 0));
}

cudaError_t launch_lmhead_logits(const void* hidden, int64_t ldh, const void* weight, int64_t ldw, int64_t n_rows,
                                 int64_t V, int64_t d, float* out, int64_t ldo, cudaStream_t st) {
    lm::LmArgs a;
    memset(&a, 0, sizeof(a));
    a.n_rows = n_rows;
    a.V = V;
    a.d = d;
    a.out = out;
    a.ldo = ldo;
    lm::schedule(a);
    CUtensorMap tA, tB;
    if (!lm::make_map(&tA, hidden, n_rows, d, ldh, lm::BM) || !lm::make_map(&tB, weight, V, d, ldw, lm::BN))
        return cudaErrorInvalidValue;
    return lm::launch_gemm<lm::StoreEpi>(tA, tB, a, st);
}

cudaError_t launch_lmhead_race(const void* hidden, int64_t ldh, const void* weight, int64_t ldw, int64_t d,
                               const RaceArgs& ra, bool verify, void* ws, cudaStream_t st) {
    lm::LmArgs a;
    memset(&a, 0, sizeof(a));
    a.n_rows = ra.n_rows;
    a.V = ra.V;
    a.d = d;
    a.key = ra.key;
    a.ctx = ra.ctx;
    a.pos = ra.pos;
    a.row_k = verify ? nullptr : ra.row_k;
    a.K = verify ? 1 : ra.K;
    a.c = ra.c;
    a.status = ra.status;
    a.partials = static_cast<lm::LmPartial*>(ws);
    lm::schedule(a);
    CUtensorMap tA, tB;
    if (!lm::make_map(&tA, hidden, a.n_rows, d, ldh, lm::BM) || !lm::make_map(&tB, weight, a.V, d, ldw, lm::BN))
        return cudaErrorInvalidValue;
    cudaError_t e = a.K <= 1 ? lm::launch_gemm<lm::RaceEpi<3>>(tA, tB, a, st)
                             : lm::launch_gemm<lm::RaceEpi<lm::kLmKP>>(tA, tB, a, st);
    if (e != cudaSuccess) return e;
    const int P = 2 * a.S;
    const unsigned blocks = (unsigned)((ra.n_rows + 3) / 4);
    if (verify)
        lm::lmhead_finish_kernel<true><<<blocks, 128, 0, st>>>(ra, a.partials, P);
    else
        lm::lmhead_finish_kernel<false><<<blocks, 128, 0, st>>>(ra, a.partials, P);
    return cudaGetLastError();
}
