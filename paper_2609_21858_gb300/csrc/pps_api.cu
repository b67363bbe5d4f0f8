// pps_api.cu -- extern "C" entry points of libpps: argument validation,
// workspace layout and launches.  Every entry point returns before launching
// anything when an argument is invalid.
#include <climits>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <atomic>
#include <mutex>

#include "pps.h"
#include "pps_internal.h"

namespace pps {

static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

size_t workspace_bytes(int64_t n_rows, int32_t n_seq) {
    return align256(kSlotBytes * (size_t)(n_rows + (int64_t)kGridMax)) + align256(sizeof(uint32_t) * 2 * (size_t)n_rows) +
           align256(sizeof(uint32_t) * (size_t)(n_seq > 0 ? n_seq : 0));
}

void workspace_carve(void* ws, int64_t n_rows, int32_t n_seq, Partial** partials, uint32_t** row_cnt,
                     uint32_t** seq_cnt) {
    char* p = static_cast<char*>(ws);
    *partials = reinterpret_cast<Partial*>(p);
    p += align256(kSlotBytes * (size_t)(n_rows + (int64_t)kGridMax));
    *row_cnt = reinterpret_cast<uint32_t*>(p);  // [n_rows] arrival counters, then [n_rows] shared row bounds
    p += align256(sizeof(uint32_t) * 2 * (size_t)n_rows);
    *seq_cnt = reinterpret_cast<uint32_t*>(p);
}

static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

static pps_status check_rows(const void* logits, pps_dtype dtype, int64_t n_rows, int64_t vocab, int64_t stride,
                             const pps_row_ids& ids, float T) {
    if (dtype != PPS_F32 && dtype != PPS_BF16) return PPS_ERR_UNSUPPORTED;
    if (n_rows < 0 || vocab < 1 || vocab > (int64_t(1) << 31) - 1 || stride < vocab) return PPS_ERR_INVALID_ARG;
    if (n_rows > 0 && (!logits || !ids.key || !ids.ctx_hash || !ids.pos)) return PPS_ERR_INVALID_ARG;
    if (!(T > 0.0f) || !std::isfinite(T)) return PPS_ERR_INVALID_ARG;
    return PPS_OK;
}

static bool vec_ok(const void* logits, pps_dtype dtype, int64_t stride) {
    size_t esz = dtype == PPS_BF16 ? 2 : 4;
    return aligned16(logits) && ((size_t)stride * esz) % 16 == 0;
}

static RaceArgs base_args(const void* logits, pps_dtype dtype, int64_t n_rows, int64_t vocab, int64_t stride,
                          const pps_row_ids& ids, float T) {
    RaceArgs a;
    std::memset(&a, 0, sizeof(a));
    a.logits = logits;
    a.n_rows = n_rows;
    a.V = vocab;
    a.stride = stride;
    a.key = ids.key;
    a.ctx = ids.ctx_hash;
    a.pos = ids.pos;
    a.T = T;
    a.c = (float)(1.4426950408889634074 / (double)T);
    int vw = dtype == PPS_BF16 ? 8 : 4;
    a.nv = (vocab + vw - 1) / vw;
    a.total = n_rows * a.nv;
    return a;
}

// ---------------------------------------------------------------- fixed scratch of the no-alloc entry point
//
// The array below is the whole scratch of pps_draft_list_noalloc: partial
// lists for PPS_NOALLOC_MAX_ROWS rows plus one per warp of a grid capped at
// PPS_NOALLOC_MAX_WARPS warps (slot = warp + row), then one arrival counter
// per row.  In host code its name is only a stand-in for the symbol, not a
// device address; the address is looked up per device with
// cudaGetSymbolAddress and cached.
constexpr size_t kNoAllocPartialBytes = sizeof(Partial) * (size_t)(PPS_NOALLOC_MAX_ROWS + PPS_NOALLOC_MAX_WARPS);
constexpr size_t kNoAllocCounterBytes = sizeof(uint32_t) * 2 * (size_t)PPS_NOALLOC_MAX_ROWS;
constexpr size_t kNoAllocScratchBytes = kNoAllocPartialBytes + kNoAllocCounterBytes;
static_assert(kNoAllocScratchBytes == PPS_NOALLOC_SCRATCH_BYTES, "pps.h states the no-alloc scratch size");
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
static std::mutex g_noalloc_mu;
static void* g_noalloc_ptr[kMaxDevices];

int device_sm_count() {
    static std::atomic<int> cache[kMaxDevices];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    int v = dev >= 0 && dev < kMaxDevices ? cache[dev].load(std::memory_order_relaxed) : 0;
    if (v == 0) {
        if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) v = 1;
        if (dev >= 0 && dev < kMaxDevices) cache[dev].store(v, std::memory_order_relaxed);
    }
    return v;
}

int resident_ctas(int slot, const void* fn, int threads) {
    static std::atomic<int> cache[kMaxDevices][kOccSlots];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    const bool cached = dev >= 0 && dev < kMaxDevices && slot >= 0 && slot < kOccSlots;
    int v = cached ? cache[dev][slot].load(std::memory_order_relaxed) : 0;
    if (v == 0) {
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, fn, threads, 0) != cudaSuccess || v <= 0) v = 1;
        if (cached) cache[dev][slot].store(v, std::memory_order_relaxed);
    }
    return v;
}

// Device address of the scratch on the current device (set up on first use).
static pps_status noalloc_scratch(void** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return PPS_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return PPS_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return PPS_ERR_CUDA;
        g_noalloc_ptr[dev] = p;
    }
    *out = g_noalloc_ptr[dev];
    return PPS_OK;
}

}  // namespace pps

using namespace pps;

extern "C" {

#define PPS_STR2(x) #x
#define PPS_STR(x) PPS_STR2(x)
const char* pps_version(void) { return "libpps 0.1 (sm_103a, Philox4x32-" PPS_STR(PPS_PHILOX_ROUNDS) ")"; }

const char* pps_status_string(pps_status s) {
    switch (s) {
        case PPS_OK: return "ok";
        case PPS_ERR_INVALID_ARG: return "invalid argument";
        case PPS_ERR_UNSUPPORTED: return "unsupported dtype or mode";
        case PPS_ERR_WORKSPACE: return "workspace missing or too small";
        case PPS_ERR_CUDA: return "CUDA launch failed";
        case PPS_ERR_SIZE: return "problem larger than the no-alloc scratch";
    }
    return "unknown status";
}

int pps_philox_rounds(void) { return PPS_PHILOX_ROUNDS; }

size_t pps_workspace_size(int64_t n_rows, int64_t vocab, int32_t K, int32_t n_seq) {
    (void)vocab;
    (void)K;
    if (n_rows < 0) n_rows = 0;
    return workspace_bytes(n_rows, n_seq);
}

pps_status pps_workspace_clear(void* ws, size_t ws_bytes, pps_stream_t stream) {
    if (!ws && ws_bytes) return PPS_ERR_INVALID_ARG;
    if (ws_bytes == 0) return PPS_OK;
    return cudaMemsetAsync(ws, 0, ws_bytes, (cudaStream_t)stream) == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

// top_k = 0: no truncation (the full-vocabulary race)
static pps_status check_trunc(int32_t top_k, float top_p) {
    if (top_k < 1 || top_k > PPS_MAX_TOP_K) return PPS_ERR_INVALID_ARG;
    if (!(top_p > 0.0f) || !(top_p <= 1.0f)) return PPS_ERR_INVALID_ARG;
    return PPS_OK;
}

static pps_status draft_list(const void* q_logits, pps_dtype dtype, int64_t n_rows, int64_t vocab, int64_t row_stride,
                             pps_row_ids ids, float temperature, int32_t top_k, float top_p, int32_t K,
                             const int32_t* row_k, pps_draft_mode mode, int32_t* out_tok, float* out_key,
                             int32_t* out_mult, int32_t* out_ndistinct, int32_t* out_samples, uint32_t* status,
                             void* ws, size_t ws_bytes, pps_stream_t stream) {
    pps_status st = check_rows(q_logits, dtype, n_rows, vocab, row_stride, ids, temperature);
    if (st != PPS_OK) return st;
    if (mode != PPS_DRAFT_DISTINCT && mode != PPS_DRAFT_IID) return PPS_ERR_UNSUPPORTED;
    if (K < 1 || K > PPS_MAX_K || K > vocab) return PPS_ERR_INVALID_ARG;
    if (n_rows == 0) return PPS_OK;
    if (!out_tok || !out_mult || !out_ndistinct) return PPS_ERR_INVALID_ARG;
    if (!ws || ws_bytes < workspace_bytes(n_rows, 0)) return PPS_ERR_WORKSPACE;
    RaceArgs a = base_args(q_logits, dtype, n_rows, vocab, row_stride, ids, temperature);
    a.K = K;
    a.row_k = row_k;
    a.iid = mode == PPS_DRAFT_IID;
    a.out_tok = out_tok;
    a.out_key = out_key;
    a.out_mult = out_mult;
    a.out_nd = out_ndistinct;
    a.out_samples = out_samples;
    a.status = status;
    workspace_carve(ws, n_rows, 0, &a.partials, &a.row_cnt, &a.seq_cnt);
    a.row_bound = a.row_cnt + n_rows;
    a.tpartials = reinterpret_cast<TruncPartial*>(a.partials);
    a.top_k = top_k;
    a.top_p = top_p;
    const int dt = dtype == PPS_BF16 ? 1 : 0;
    const bool vec = vec_ok(q_logits, dtype, row_stride);
    cudaError_t e;
    if (top_k > 0) {
        a.G = trunc_grid(a.total, a.n_rows, dt, false, vec);
        e = launch_trunc(a, dt, false, vec, (cudaStream_t)stream);
    } else {
        a.G = race_grid(a.total, dt, false, vec, false, a.n_rows);
        e = launch_race(a, dt, false, vec, (cudaStream_t)stream);
    }
    return e == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

pps_status pps_draft_list(const void* q_logits, pps_dtype dtype, int64_t n_rows, int64_t vocab, int64_t row_stride,
                          pps_row_ids ids, float temperature, int32_t K, const int32_t* row_k, pps_draft_mode mode,
                          int32_t* out_tok, float* out_key, int32_t* out_mult, int32_t* out_ndistinct,
                          int32_t* out_samples, uint32_t* status, void* ws, size_t ws_bytes, pps_stream_t stream) {
    return draft_list(q_logits, dtype, n_rows, vocab, row_stride, ids, temperature, 0, 1.0f, K, row_k, mode, out_tok,
                      out_key, out_mult, out_ndistinct, out_samples, status, ws, ws_bytes, stream);
}

pps_status pps_draft_list_trunc(const void* q_logits, pps_dtype dtype, int64_t n_rows, int64_t vocab,
                                int64_t row_stride, pps_row_ids ids, float temperature, int32_t top_k, float top_p,
                                int32_t K, const int32_t* row_k, pps_draft_mode mode, int32_t* out_tok,
                                float* out_key, int32_t* out_mult, int32_t* out_ndistinct, int32_t* out_samples,
                                uint32_t* status, void* ws, size_t ws_bytes, pps_stream_t stream) {
    pps_status st = check_trunc(top_k, top_p);
    if (st != PPS_OK) return st;
    return draft_list(q_logits, dtype, n_rows, vocab, row_stride, ids, temperature, top_k, top_p, K, row_k, mode,
                      out_tok, out_key, out_mult, out_ndistinct, out_samples, status, ws, ws_bytes, stream);
}

static pps_status verify_tree(const void* p_logits, pps_dtype dtype, int64_t n_nodes, int64_t vocab,
                              int64_t row_stride, pps_row_ids ids, float temperature, int32_t top_k, float top_p,
                              int32_t n_seq, int32_t gamma, const int32_t* seq_off, const int32_t* node_draft_row,
                              int64_t n_draft, const int32_t* draft_tok, const int32_t* draft_ndistinct, int32_t K,
                              const int32_t* child_node, int32_t* out_winner, uint32_t* out_word,
                              int32_t* out_accept_len, int32_t* out_n_emitted, int32_t* out_emitted, float* out_score,
                              double* out_score_sum, uint32_t* status, void* ws, size_t ws_bytes,
                              pps_stream_t stream) {
    pps_status st = check_rows(p_logits, dtype, n_nodes, vocab, row_stride, ids, temperature);
    if (st != PPS_OK) return st;
    if (n_seq < 0 || gamma < 1 || gamma > 64 || K < 1 || K > PPS_MAX_K || n_draft < 0) return PPS_ERR_INVALID_ARG;
    if (n_nodes == 0 || n_seq == 0) return n_nodes == 0 && n_seq == 0 ? PPS_OK : PPS_ERR_INVALID_ARG;
    if (n_nodes < n_seq) return PPS_ERR_INVALID_ARG;
    if (!seq_off || !node_draft_row || !draft_tok || !draft_ndistinct || !child_node || !out_winner || !out_word ||
        !out_accept_len || !out_n_emitted || !out_emitted || !out_score || !out_score_sum)
        return PPS_ERR_INVALID_ARG;
    if (!ws || ws_bytes < workspace_bytes(n_nodes, n_seq)) return PPS_ERR_WORKSPACE;
    RaceArgs a = base_args(p_logits, dtype, n_nodes, vocab, row_stride, ids, temperature);
    a.K = 1;
    a.n_seq = n_seq;
    a.gamma = gamma;
    a.seq_off = seq_off;
    a.node_draft_row = node_draft_row;
    a.n_draft = n_draft;
    a.draft_tok = draft_tok;
    a.draft_nd = draft_ndistinct;
    a.Kd = K;
    a.child_node = child_node;
    a.out_winner = out_winner;
    a.out_word = out_word;
    a.out_acc = out_accept_len;
    a.out_ne = out_n_emitted;
    a.out_em = out_emitted;
    a.out_sc = out_score;
    a.out_ss = out_score_sum;
    a.status = status;
    workspace_carve(ws, n_nodes, n_seq, &a.partials, &a.row_cnt, &a.seq_cnt);
    a.row_bound = a.row_cnt + n_nodes;
    a.tpartials = reinterpret_cast<TruncPartial*>(a.partials);
    a.top_k = top_k;
    a.top_p = top_p;
    const int dt = dtype == PPS_BF16 ? 1 : 0;
    const bool vec = vec_ok(p_logits, dtype, row_stride);
    cudaError_t e;
    if (top_k > 0) {
        a.G = trunc_grid(a.total, a.n_rows, dt, true, vec);
        e = launch_trunc(a, dt, true, vec, (cudaStream_t)stream);
    } else {
        a.G = race_grid(a.total, dt, true, vec, false, a.n_rows);
        e = launch_race(a, dt, true, vec, (cudaStream_t)stream);
    }
    return e == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

pps_status pps_verify_tree(const void* p_logits, pps_dtype dtype, int64_t n_nodes, int64_t vocab, int64_t row_stride,
                           pps_row_ids ids, float temperature, int32_t n_seq, int32_t gamma, const int32_t* seq_off,
                           const int32_t* node_draft_row, int64_t n_draft, const int32_t* draft_tok,
                           const int32_t* draft_ndistinct, int32_t K, const int32_t* child_node, int32_t* out_winner,
                           uint32_t* out_word, int32_t* out_accept_len, int32_t* out_n_emitted, int32_t* out_emitted,
                           float* out_score, double* out_score_sum, uint32_t* status, void* ws, size_t ws_bytes,
                           pps_stream_t stream) {
    return verify_tree(p_logits, dtype, n_nodes, vocab, row_stride, ids, temperature, 0, 1.0f, n_seq, gamma, seq_off,
                       node_draft_row, n_draft, draft_tok, draft_ndistinct, K, child_node, out_winner, out_word,
                       out_accept_len, out_n_emitted, out_emitted, out_score, out_score_sum, status, ws, ws_bytes,
                       stream);
}

pps_status pps_verify_tree_trunc(const void* p_logits, pps_dtype dtype, int64_t n_nodes, int64_t vocab,
                                 int64_t row_stride, pps_row_ids ids, float temperature, int32_t top_k, float top_p,
                                 int32_t n_seq, int32_t gamma, const int32_t* seq_off, const int32_t* node_draft_row,
                                 int64_t n_draft, const int32_t* draft_tok, const int32_t* draft_ndistinct, int32_t K,
                                 const int32_t* child_node, int32_t* out_winner, uint32_t* out_word,
                                 int32_t* out_accept_len, int32_t* out_n_emitted, int32_t* out_emitted,
                                 float* out_score, double* out_score_sum, uint32_t* status, void* ws,
                                 size_t ws_bytes, pps_stream_t stream) {
    pps_status st = check_trunc(top_k, top_p);
    if (st != PPS_OK) return st;
    return verify_tree(p_logits, dtype, n_nodes, vocab, row_stride, ids, temperature, top_k, top_p, n_seq, gamma,
                       seq_off, node_draft_row, n_draft, draft_tok, draft_ndistinct, K, child_node, out_winner,
                       out_word, out_accept_len, out_n_emitted, out_emitted, out_score, out_score_sum, status, ws,
                       ws_bytes, stream);
}

pps_status pps_draft_list_noalloc(const void* q_logits, pps_dtype dtype, int64_t n_rows, int64_t vocab,
                                  int64_t row_stride, pps_row_ids ids, float temperature, int32_t K,
                                  const int32_t* row_k, pps_draft_mode mode, int32_t* out_tok, float* out_key,
                                  int32_t* out_mult, int32_t* out_ndistinct, int32_t* out_samples, uint32_t* status,
                                  pps_stream_t stream) {
    pps_status st = check_rows(q_logits, dtype, n_rows, vocab, row_stride, ids, temperature);
    if (st != PPS_OK) return st;
    if (mode != PPS_DRAFT_DISTINCT && mode != PPS_DRAFT_IID) return PPS_ERR_UNSUPPORTED;
    if (K < 1 || K > PPS_MAX_K || K > vocab) return PPS_ERR_INVALID_ARG;
    if (n_rows == 0) return PPS_OK;
    if (!out_tok || !out_mult || !out_ndistinct) return PPS_ERR_INVALID_ARG;
    if (n_rows > PPS_NOALLOC_MAX_ROWS) return PPS_ERR_SIZE;
    void* scratch = nullptr;
    st = noalloc_scratch(&scratch);
    if (st != PPS_OK) return st;
    char* base = static_cast<char*>(scratch);
    uint32_t* row_cnt = reinterpret_cast<uint32_t*>(base + kNoAllocPartialBytes);
    // the arrival counters and shared row bounds must start at zero; the partial lists need no clearing
    if (cudaMemsetAsync(row_cnt, 0, sizeof(uint32_t) * 2 * (size_t)n_rows, (cudaStream_t)stream) != cudaSuccess)
        return PPS_ERR_CUDA;
    RaceArgs a = base_args(q_logits, dtype, n_rows, vocab, row_stride, ids, temperature);
    a.K = K;
    a.row_k = row_k;
    a.iid = mode == PPS_DRAFT_IID;
    a.out_tok = out_tok;
    a.out_key = out_key;
    a.out_mult = out_mult;
    a.out_nd = out_ndistinct;
    a.out_samples = out_samples;
    a.status = status;
    a.partials = reinterpret_cast<Partial*>(base);
    a.row_cnt = row_cnt;
    a.row_bound = row_cnt + n_rows;
    a.seq_cnt = nullptr;
    const int dt = dtype == PPS_BF16 ? 1 : 0;
    const bool vec = vec_ok(q_logits, dtype, row_stride);
    a.G = race_grid(a.total, dt, false, vec, false, a.n_rows);
    if (a.G > PPS_NOALLOC_MAX_WARPS) a.G = PPS_NOALLOC_MAX_WARPS;
    return launch_race(a, dt, false, vec, (cudaStream_t)stream) == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

// ---------------------------------------------------------------- LM head

static pps_status check_lmhead(const void* hidden, int64_t ldh, const void* weight, int64_t ldw, int64_t n_rows,
                               int64_t vocab, int64_t d) {
    if (n_rows < 0 || n_rows > INT32_MAX || vocab < 1 || vocab > INT32_MAX || d < 1 || ldh < d || ldw < d)
        return PPS_ERR_INVALID_ARG;
    if (!weight || (n_rows > 0 && !hidden)) return PPS_ERR_INVALID_ARG;
    // TMA: 16-byte aligned bases and 16-byte row strides
    if (!aligned16(weight) || (hidden && !aligned16(hidden)) || ldh % 8 != 0 || ldw % 8 != 0) return PPS_ERR_INVALID_ARG;
    return PPS_OK;
}

size_t pps_lmhead_workspace_size(int64_t n_rows, int32_t n_seq) {
    return lmhead_workspace_bytes(n_rows < 0 ? 0 : n_rows, n_seq);
}

pps_status pps_lmhead_logits(const void* hidden, int64_t ld_hidden, const void* weight, int64_t ld_weight,
                             int64_t n_rows, int64_t vocab, int64_t d, float* out_logits, int64_t ld_out,
                             pps_stream_t stream) {
    pps_status st = check_lmhead(hidden, ld_hidden, weight, ld_weight, n_rows, vocab, d);
    if (st != PPS_OK) return st;
    if (ld_out < vocab || (n_rows > 0 && !out_logits)) return PPS_ERR_INVALID_ARG;
    if (n_rows == 0) return PPS_OK;
    return launch_lmhead_logits(hidden, ld_hidden, weight, ld_weight, n_rows, vocab, d, out_logits, ld_out,
                                (cudaStream_t)stream) == cudaSuccess
               ? PPS_OK
               : PPS_ERR_CUDA;
}

pps_status pps_lmhead_draft_list(const void* hidden, int64_t ld_hidden, const void* weight, int64_t ld_weight,
                                 int64_t n_rows, int64_t vocab, int64_t d, pps_row_ids ids, float temperature,
                                 int32_t K, const int32_t* row_k, pps_draft_mode mode, int32_t* out_tok,
                                 float* out_key, int32_t* out_mult, int32_t* out_ndistinct, int32_t* out_samples,
                                 uint32_t* status, void* ws, size_t ws_bytes, pps_stream_t stream) {
    pps_status st = check_lmhead(hidden, ld_hidden, weight, ld_weight, n_rows, vocab, d);
    if (st != PPS_OK) return st;
    if (!(temperature > 0.0f) || !std::isfinite(temperature)) return PPS_ERR_INVALID_ARG;
    if (n_rows > 0 && (!ids.key || !ids.ctx_hash || !ids.pos)) return PPS_ERR_INVALID_ARG;
    if (mode != PPS_DRAFT_DISTINCT && mode != PPS_DRAFT_IID) return PPS_ERR_UNSUPPORTED;
    if (K < 1 || K > PPS_LMHEAD_MAX_K || K > vocab) return PPS_ERR_INVALID_ARG;
    if (n_rows == 0) return PPS_OK;
    if (!out_tok || !out_mult || !out_ndistinct) return PPS_ERR_INVALID_ARG;
    if (!ws || ws_bytes < lmhead_workspace_bytes(n_rows, 0)) return PPS_ERR_WORKSPACE;
    RaceArgs a = base_args(nullptr, PPS_F32, n_rows, vocab, vocab, ids, temperature);
    a.K = K;
    a.row_k = row_k;
    a.iid = mode == PPS_DRAFT_IID;
    a.out_tok = out_tok;
    a.out_key = out_key;
    a.out_mult = out_mult;
    a.out_nd = out_ndistinct;
    a.out_samples = out_samples;
    a.status = status;
    return launch_lmhead_race(hidden, ld_hidden, weight, ld_weight, d, a, false, ws, (cudaStream_t)stream) ==
                   cudaSuccess
               ? PPS_OK
               : PPS_ERR_CUDA;
}

pps_status pps_lmhead_verify_tree(const void* hidden, int64_t ld_hidden, const void* weight, int64_t ld_weight,
                                  int64_t n_nodes, int64_t vocab, int64_t d, pps_row_ids ids, float temperature,
                                  int32_t n_seq, int32_t gamma, const int32_t* seq_off, const int32_t* node_draft_row,
                                  int64_t n_draft, const int32_t* draft_tok, const int32_t* draft_ndistinct,
                                  int32_t K, const int32_t* child_node, int32_t* out_winner, uint32_t* out_word,
                                  int32_t* out_accept_len, int32_t* out_n_emitted, int32_t* out_emitted,
                                  float* out_score, double* out_score_sum, uint32_t* status, void* ws,
                                  size_t ws_bytes, pps_stream_t stream) {
    pps_status st = check_lmhead(hidden, ld_hidden, weight, ld_weight, n_nodes, vocab, d);
    if (st != PPS_OK) return st;
    if (!(temperature > 0.0f) || !std::isfinite(temperature)) return PPS_ERR_INVALID_ARG;
    if (n_seq < 0 || gamma < 1 || gamma > 64 || K < 1 || K > PPS_MAX_K || n_draft < 0) return PPS_ERR_INVALID_ARG;
    if (n_nodes == 0 || n_seq == 0) return n_nodes == 0 && n_seq == 0 ? PPS_OK : PPS_ERR_INVALID_ARG;
    if (n_nodes < n_seq) return PPS_ERR_INVALID_ARG;
    if (!ids.key || !ids.ctx_hash || !ids.pos) return PPS_ERR_INVALID_ARG;
    if (!seq_off || !node_draft_row || !draft_tok || !draft_ndistinct || !child_node || !out_winner || !out_word ||
        !out_accept_len || !out_n_emitted || !out_emitted || !out_score || !out_score_sum)
        return PPS_ERR_INVALID_ARG;
    const size_t need = lmhead_workspace_bytes(n_nodes, n_seq);
    if (!ws || ws_bytes < need) return PPS_ERR_WORKSPACE;
    RaceArgs a = base_args(nullptr, PPS_F32, n_nodes, vocab, vocab, ids, temperature);
    a.K = 1;
    a.n_seq = n_seq;
    a.gamma = gamma;
    a.seq_off = seq_off;
    a.node_draft_row = node_draft_row;
    a.n_draft = n_draft;
    a.draft_tok = draft_tok;
    a.draft_nd = draft_ndistinct;
    a.Kd = K;
    a.child_node = child_node;
    a.out_winner = out_winner;
    a.out_word = out_word;
    a.out_acc = out_accept_len;
    a.out_ne = out_n_emitted;
    a.out_em = out_emitted;
    a.out_sc = out_score;
    a.out_ss = out_score_sum;
    a.status = status;
    // the sequence tickets follow the partial lists
    a.seq_cnt = reinterpret_cast<uint32_t*>(static_cast<char*>(ws) + lmhead_workspace_bytes(n_nodes, 0));
    return launch_lmhead_race(hidden, ld_hidden, weight, ld_weight, d, a, true, ws, (cudaStream_t)stream) ==
                   cudaSuccess
               ? PPS_OK
               : PPS_ERR_CUDA;
}

pps_status pps_wm_detect(const int32_t* tokens, pps_row_ids ids, int64_t n, int32_t n_seg, const int64_t* seg_off,
                         pps_score_kind kind, double param, float* out_score, double* out_sum, double* out_logp,
                         pps_stream_t stream) {
    if (n < 0) return PPS_ERR_INVALID_ARG;
    if (seg_off && n_seg < 1) return PPS_ERR_INVALID_ARG;
    if (n > 0 && (!tokens || !ids.key || !ids.ctx_hash || !ids.pos)) return PPS_ERR_INVALID_ARG;
    if (!out_score && !out_sum) return PPS_ERR_INVALID_ARG;
    if (out_logp && !out_sum) return PPS_ERR_INVALID_ARG;
    ScoreParams P;
    std::memset(&P, 0, sizeof(P));
    P.kind = (int)kind;
    switch (kind) {
        case PPS_SCORE_AARONSON:
        case PPS_SCORE_U:
            break;
        case PPS_SCORE_LI: {
            if (!(param > 0.0 && param < 1.0)) return PPS_ERR_INVALID_ARG;
            const double k = std::floor(1.0 / (1.0 - param)), q = 1.0 - k * (1.0 - param);
            P.k = (float)k;
            P.a = (float)(param / (1.0 - param));
            P.has_q = q > 0.0 ? 1.0f : 0.0f;
            P.b = q > 0.0 ? (float)((1.0 - q) / q) : 0.0f;
            break;
        }
        case PPS_SCORE_POWER_LAW:
            if (!(param > 0.0 && param <= 1.0)) return PPS_ERR_INVALID_ARG;
            P.cap = (float)(1.0 / std::sqrt(param));
            P.centre = (float)(2.0 - std::sqrt(param));
            break;
        default:
            return PPS_ERR_UNSUPPORTED;
    }
    cudaError_t e = launch_wm_score(tokens, ids.key, ids.ctx_hash, ids.pos, n, seg_off ? n_seg : 1, seg_off, P,
                                    out_score, out_sum, out_logp, (cudaStream_t)stream);
    return e == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

pps_status pps_wm_score(const int32_t* tokens, pps_row_ids ids, int64_t n, int32_t n_seg, const int64_t* seg_off,
                        float* out_score, double* out_sum, pps_stream_t stream) {
    return pps_wm_detect(tokens, ids, n, n_seg, seg_off, PPS_SCORE_AARONSON, 0.0, out_score, out_sum, nullptr, stream);
}

pps_status pps_tree_expand(int32_t n_seq, int32_t K, int32_t gamma, int32_t depth, const int32_t* draft_tok,
                           const int32_t* draft_mult, const int32_t* draft_ndistinct, pps_row_ids rows,
                           const int32_t* row_k, uint64_t* next_key, uint64_t* next_ctx, uint32_t* next_pos,
                           int32_t* next_k, int32_t* child_node, uint64_t* node_key, uint64_t* node_ctx,
                           uint32_t* node_pos, pps_stream_t stream) {
    if (n_seq < 0 || K < 1 || K > PPS_MAX_K || gamma < 1 || gamma > 64 || depth < 0 || depth >= gamma)
        return PPS_ERR_INVALID_ARG;
    if (n_seq == 0) return PPS_OK;
    if (!draft_tok || !draft_mult || !draft_ndistinct || !rows.key || !rows.ctx_hash || !rows.pos || !row_k ||
        !next_key || !next_ctx || !next_pos || !next_k || !child_node || !node_key || !node_ctx || !node_pos)
        return PPS_ERR_INVALID_ARG;
    cudaError_t e = launch_tree_expand(n_seq, K, gamma, depth, draft_tok, draft_mult, draft_ndistinct, rows.key,
                                       rows.ctx_hash, rows.pos, row_k, next_key, next_ctx, next_pos, next_k,
                                       child_node, node_key, node_ctx, node_pos, (cudaStream_t)stream);
    return e == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

static pps_status draft_hetero(const void* q_logits, pps_dtype dtype, int64_t n_rows, int64_t vocab,
                               int64_t row_stride, pps_row_ids ids, float temperature, int32_t top_k, float top_p,
                               const int32_t* row_block, int32_t n_blocks, int32_t* out_tok, float* out_key,
                               uint32_t* status, void* ws, size_t ws_bytes, pps_stream_t stream) {
    pps_status st = check_rows(q_logits, dtype, n_rows, vocab, row_stride, ids, temperature);
    if (st != PPS_OK) return st;
    if (n_blocks < 1 || n_blocks > PPS_MAX_BLOCKS) return PPS_ERR_INVALID_ARG;
    if (n_rows == 0) return PPS_OK;
    if (!out_tok || !row_block) return PPS_ERR_INVALID_ARG;
    if (!ws || ws_bytes < workspace_bytes(n_rows, 0)) return PPS_ERR_WORKSPACE;
    RaceArgs a = base_args(q_logits, dtype, n_rows, vocab, row_stride, ids, temperature);
    a.K = 1;
    a.out_tok = out_tok;
    a.out_key = out_key;
    a.status = status;
    // one block is the plain race (E_(i,0) = E'_i)
    if (n_blocks > 1) {
        a.row_block = row_block;
        a.n_blocks = n_blocks;
    }
    workspace_carve(ws, n_rows, 0, &a.partials, &a.row_cnt, &a.seq_cnt);
    a.row_bound = a.row_cnt + n_rows;
    a.tpartials = reinterpret_cast<TruncPartial*>(a.partials);
    a.top_k = top_k;
    a.top_p = top_p;
    const int dt = dtype == PPS_BF16 ? 1 : 0;
    const bool vec = vec_ok(q_logits, dtype, row_stride);
    cudaError_t e;
    if (top_k > 0) {
        a.G = trunc_grid(a.total, a.n_rows, dt, false, vec, n_blocks > 1);
        e = launch_trunc(a, dt, false, vec, (cudaStream_t)stream);
    } else {
        a.G = race_grid(a.total, dt, false, vec, n_blocks > 1, a.n_rows);
        e = launch_race(a, dt, false, vec, (cudaStream_t)stream);
    }
    return e == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

pps_status pps_draft_hetero(const void* q_logits, pps_dtype dtype, int64_t n_rows, int64_t vocab, int64_t row_stride,
                            pps_row_ids ids, float temperature, const int32_t* row_block, int32_t n_blocks,
                            int32_t* out_tok, float* out_key, uint32_t* status, void* ws, size_t ws_bytes,
                            pps_stream_t stream) {
    return draft_hetero(q_logits, dtype, n_rows, vocab, row_stride, ids, temperature, 0, 1.0f, row_block, n_blocks,
                        out_tok, out_key, status, ws, ws_bytes, stream);
}

pps_status pps_draft_hetero_trunc(const void* q_logits, pps_dtype dtype, int64_t n_rows, int64_t vocab,
                                  int64_t row_stride, pps_row_ids ids, float temperature, int32_t top_k, float top_p,
                                  const int32_t* row_block, int32_t n_blocks, int32_t* out_tok, float* out_key,
                                  uint32_t* status, void* ws, size_t ws_bytes, pps_stream_t stream) {
    pps_status st = check_trunc(top_k, top_p);
    if (st != PPS_OK) return st;
    return draft_hetero(q_logits, dtype, n_rows, vocab, row_stride, ids, temperature, top_k, top_p, row_block,
                        n_blocks, out_tok, out_key, status, ws, ws_bytes, stream);
}

pps_status pps_hetero_expand(int32_t n_seq, int32_t n_blocks, int32_t gamma, int32_t depth, const int32_t* draft_tok,
                             pps_row_ids rows, const int32_t* row_owner, uint64_t* next_key, uint64_t* next_ctx,
                             uint32_t* next_pos, int32_t* next_owner, int32_t* list_tok, int32_t* list_ndistinct,
                             int32_t* child_node, uint64_t* node_key, uint64_t* node_ctx, uint32_t* node_pos,
                             pps_stream_t stream) {
    if (n_seq < 0 || n_blocks < 1 || n_blocks > PPS_MAX_BLOCKS || gamma < 1 || gamma > 64 || depth < 0 ||
        depth >= gamma)
        return PPS_ERR_INVALID_ARG;
    if (n_seq == 0) return PPS_OK;
    if (!draft_tok || !rows.key || !rows.ctx_hash || !rows.pos || !row_owner || !list_tok || !list_ndistinct ||
        !child_node || !node_key || !node_ctx || !node_pos)
        return PPS_ERR_INVALID_ARG;
    if (depth + 1 < gamma && (!next_key || !next_ctx || !next_pos || !next_owner)) return PPS_ERR_INVALID_ARG;
    cudaError_t e = launch_hetero_expand(n_seq, n_blocks, gamma, depth, draft_tok, rows.key, rows.ctx_hash, rows.pos,
                                         row_owner, next_key, next_ctx, next_pos, next_owner, list_tok,
                                         list_ndistinct, child_node, node_key, node_ctx, node_pos,
                                         (cudaStream_t)stream);
    return e == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

pps_status pps_hetero_block(const int32_t* tokens, pps_row_ids ids, int64_t n, int32_t n_blocks, int32_t* out_block,
                            pps_stream_t stream) {
    if (n < 0 || n_blocks < 1 || n_blocks > PPS_MAX_BLOCKS) return PPS_ERR_INVALID_ARG;
    if (n == 0) return PPS_OK;
    if (!tokens || !ids.key || !ids.ctx_hash || !ids.pos || !out_block) return PPS_ERR_INVALID_ARG;
    cudaError_t e = launch_hetero_block(n, n_blocks, tokens, ids.key, ids.ctx_hash, ids.pos, out_block,
                                        (cudaStream_t)stream);
    return e == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

pps_status pps_philox_words(pps_row_ids ids, int64_t n_rows, int64_t vocab, int32_t arrival, uint32_t* out,
                            pps_stream_t stream) {
    if (n_rows < 0 || vocab < 1 || arrival < 1) return PPS_ERR_INVALID_ARG;
    if (n_rows > 0 && (!ids.key || !ids.ctx_hash || !ids.pos || !out)) return PPS_ERR_INVALID_ARG;
    cudaError_t e = launch_words(ids.key, ids.ctx_hash, ids.pos, n_rows, vocab, arrival, out, (cudaStream_t)stream);
    return e == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

pps_status pps_selftest_key_error(uint64_t w_begin, uint64_t w_end, float* out_max_err, pps_stream_t stream) {
    if (!out_max_err || w_end > (uint64_t(1) << 32) || w_begin > w_end) return PPS_ERR_INVALID_ARG;
    return launch_selftest(w_begin, w_end, out_max_err, (cudaStream_t)stream) == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

pps_status pps_selftest_lg2_error(float x_lo, float x_hi, float* out_max_err, pps_stream_t stream) {
    if (!out_max_err || !(x_lo > 0.0f) || !(x_hi >= x_lo) || !std::isfinite(x_hi)) return PPS_ERR_INVALID_ARG;
    uint32_t b0, b1;
    std::memcpy(&b0, &x_lo, 4);
    std::memcpy(&b1, &x_hi, 4);
    return launch_selftest_lg2(b0, b1, out_max_err, (cudaStream_t)stream) == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

pps_status pps_selftest_philox_rate(uint64_t n_blocks, uint32_t* out, int32_t out_len, pps_stream_t stream) {
    if (!out || out_len < 256 || n_blocks == 0) return PPS_ERR_INVALID_ARG;
    return launch_philox_rate(n_blocks, out, out_len, (cudaStream_t)stream) == cudaSuccess ? PPS_OK : PPS_ERR_CUDA;
}

}  // extern "C"
