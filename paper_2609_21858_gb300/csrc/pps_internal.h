// pps_internal.h -- host/device structures shared by the libpps translation units.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

// Rounds of the keyed source's Philox4x32 (pps_device.cuh): 10 unless the
// library is built with -DPPS_PHILOX_ROUNDS=7 (libpps_r7.so).
#ifndef PPS_PHILOX_ROUNDS
#define PPS_PHILOX_ROUNDS 10
#endif

namespace pps {

constexpr int kThreads = 32;            // one warp per CTA: per-row values are CTA-uniform
constexpr int kWarps = kThreads / 32;
constexpr int kGridMax = 16384;         // upper bound on the streaming grid (one-warp CTAs)
constexpr int64_t kMinVecsPerWarp = 256;  // 16-byte vectors per warp below which the grid shrinks

// one partial candidate list of a row segment (sorted ascending by (key, idx))
struct alignas(16) Partial {
    float key[32];
    int32_t idx[32];
    float theta_drop;  // every token of the segment left out has an fp32 key >= theta_drop
    int32_t n;
    int32_t pad[2];
};

// one partial top-k list of a row segment for the truncated race (sorted by
// logit descending, then token ascending; empty entries (-inf, INT_MAX))
constexpr int kTopMax = 64;  // largest top-k of the truncated race
struct alignas(16) TruncPartial {
    float v[kTopMax];
    int32_t idx[kTopMax];
    float dropmax;  // largest logit evicted from the segment's list (-inf: none)
    int32_t pad[3];
};
// workspace slot: room for either kind of partial list
constexpr size_t kSlotBytes = sizeof(TruncPartial) > sizeof(Partial) ? sizeof(TruncPartial) : sizeof(Partial);

struct RaceArgs {
    const void* logits;
    int64_t n_rows, V, stride;
    const uint64_t* key;
    const uint64_t* ctx;
    const uint32_t* pos;
    float T;  // temperature
    float c;  // log2(e) / T
    // draft side
    int K;
    const int32_t* row_k;
    int iid;
    int32_t* out_tok;
    float* out_key;
    int32_t* out_mult;
    int32_t* out_nd;
    int32_t* out_samples;
    // target side + walk
    int n_seq, gamma;
    const int32_t* seq_off;
    const int32_t* node_draft_row;
    int64_t n_draft;
    const int32_t* draft_tok;
    const int32_t* draft_nd;
    int Kd;
    const int32_t* child_node;
    int32_t* out_winner;
    uint32_t* out_word;
    int32_t* out_acc;
    int32_t* out_ne;
    int32_t* out_em;
    float* out_sc;
    double* out_ss;
    uint32_t* status;
    // partition of the flattened (row, vector) range over the grid
    int64_t nv;     // 16-byte vectors per row (last one may be partial)
    int64_t total;  // n_rows * nv
    int G;
    // proposal rows of the augmented race (draft side only; row_block NULL = off):
    // row r is proposal row_block[r] of n_blocks
    const int32_t* row_block;
    int n_blocks;
    // truncation (truncated race only): top-k in [1, kTopMax], top-p in (0, 1]
    int top_k;
    float top_p;
    // workspace
    Partial* partials;   // [n_rows + kGridMax]: slot (warp + row)
    TruncPartial* tpartials;  // the same slots, for the truncated race
    uint32_t* row_cnt;   // [n_rows]
    uint32_t* row_bound; // [n_rows] shared filter bound of a row cut between warps (0 = none)
    uint32_t* seq_cnt;   // [n_seq]
};

// Programmatic dependent launch.  A kernel launched with launch_pdl may start
// while the previous kernel on its stream drains; it calls pdl_wait() before it
// reads anything a previous kernel wrote (the wait returns once that kernel has
// completed and its memory is visible; without the attribute it is a no-op) and
// pdl_launch_dependents() to let the next kernel start launching in turn.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... Args, typename... Act>
inline cudaError_t launch_pdl(void (*kernel)(Args...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                              Act&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Act&&>(args)...);
}

size_t workspace_bytes(int64_t n_rows, int32_t n_seq);
void workspace_carve(void* ws, int64_t n_rows, int32_t n_seq, Partial** partials, uint32_t** row_cnt,
                     uint32_t** seq_cnt);

// launchers (pps_race.cu)
// Launch limits of the current device, cached per device on first use (relaxed
// atomics: concurrent first calls from several host threads store the same value).
// resident_ctas: CTAs of `threads` threads of kernel `fn` resident per SM; `slot`
// (< kOccSlots) names the kernel in the cache.
constexpr int kOccSlots = 32;
constexpr int kOccRace = 0;    // 12 slots: dtype x (draft, verify, block) x vec
constexpr int kOccTrunc = 12;  // 12 slots, the same
constexpr int kOccScore = 24;
int device_sm_count();
int resident_ctas(int slot, const void* fn, int threads);

cudaError_t launch_race(const RaceArgs& a, int dtype, bool verify, bool vec, cudaStream_t stream);
int race_grid(int64_t total, int dtype, bool verify, bool vec, bool blk = false, int64_t n_rows = 0);
cudaError_t launch_trunc(const RaceArgs& a, int dtype, bool verify, bool vec, cudaStream_t stream);
int trunc_grid(int64_t total, int64_t n_rows, int dtype, bool verify, bool vec, bool blk = false);

// the LM-head GEMM with the race in its epilogue (pps_lmhead.cuh, in pps_race.cu).
// hidden [n_rows, d] and weight [V, d] are bf16 with row strides ldh, ldw elements.
size_t lmhead_workspace_bytes(int64_t n_rows, int32_t n_seq);
cudaError_t launch_lmhead_logits(const void* hidden, int64_t ldh, const void* weight, int64_t ldw, int64_t n_rows,
                                 int64_t V, int64_t d, float* out, int64_t ldo, cudaStream_t st);
cudaError_t launch_lmhead_race(const void* hidden, int64_t ldh, const void* weight, int64_t ldw, int64_t d,
                               const RaceArgs& ra, bool verify, void* ws, cudaStream_t st);

// launchers (pps_misc.cu)
// detection score kind and its constants (pps_device.cuh score_kind32)
struct ScoreParams {
    int kind;  // 0 Aaronson, 1 U, 2 Li, 3 power law
    float a, b, k, has_q, cap, centre;
};
cudaError_t launch_wm_score(const int32_t* tokens, const uint64_t* key, const uint64_t* ctx, const uint32_t* pos,
                            int64_t n, int32_t n_seg, const int64_t* seg_off, const ScoreParams& P, float* out_score,
                            double* out_sum, double* out_logp, cudaStream_t stream);
cudaError_t launch_tree_expand(int32_t n_seq, int32_t K, int32_t gamma, int32_t depth, const int32_t* tok,
                               const int32_t* mult, const int32_t* ndist, const uint64_t* key, const uint64_t* ctx,
                               const uint32_t* pos, const int32_t* row_k, uint64_t* next_key, uint64_t* next_ctx,
                               uint32_t* next_pos, int32_t* next_k, int32_t* child_node, uint64_t* node_key,
                               uint64_t* node_ctx, uint32_t* node_pos, cudaStream_t stream);
cudaError_t launch_hetero_expand(int32_t n_seq, int32_t B, int32_t gamma, int32_t depth, const int32_t* tok,
                                 const uint64_t* key, const uint64_t* ctx, const uint32_t* pos, const int32_t* owner,
                                 uint64_t* next_key, uint64_t* next_ctx, uint32_t* next_pos, int32_t* next_owner,
                                 int32_t* list_tok, int32_t* list_nd, int32_t* child_node, uint64_t* node_key,
                                 uint64_t* node_ctx, uint32_t* node_pos, cudaStream_t stream);
cudaError_t launch_hetero_block(int64_t n, int32_t B, const int32_t* tok, const uint64_t* key, const uint64_t* ctx,
                                const uint32_t* pos, int32_t* out, cudaStream_t stream);
cudaError_t launch_words(const uint64_t* key, const uint64_t* ctx, const uint32_t* pos, int64_t n_rows, int64_t V,
                         int32_t arrival, uint32_t* out, cudaStream_t stream);
cudaError_t launch_selftest(uint64_t w_begin, uint64_t w_end, float* out, cudaStream_t stream);
cudaError_t launch_selftest_lg2(uint32_t b0, uint32_t b1, float* out, cudaStream_t stream);
cudaError_t launch_philox_rate(uint64_t n_blocks, uint32_t* out, int out_len, cudaStream_t stream);

}  // namespace pps
