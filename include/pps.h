/*
 * pps.h -- C ABI of libpps, the GB300 (sm_103a) implementation of the keyed
 * Poisson-race multi-draft speculative sampler of "Watermarkable Multi-Draft
 * Speculative Sampling via Poisson Processes".
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Every pointer argument is DEVICE memory on the current CUDA device, owned
 *   by the caller, unless the comment says otherwise.  The library never
 *   allocates device memory and keeps no state between calls.
 * - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy default
 *   stream).  A non-PPS_OK return from argument validation is synchronous and
 *   launches nothing.  PPS_ERR_CUDA reports a failed launch (cudaGetLastError
 *   after the launch); the CUDA error itself stays readable through the CUDA
 *   runtime.  Outputs are undefined unless the call returned PPS_OK.
 * - Logits rows are `row_stride` elements apart (row_stride >= vocab),
 *   row-major, fp32 or bf16.  Rows whose start is 16-byte aligned are
 *   streamed with 128-bit loads; other layouts take a slower scalar path.
 * - Row identities (pps_row_ids) label the keyed Poisson source G(k, c) of the
 *   paper (Sec. 3.3, Alg. 3 and 4, detector algorithm of App. E): a 64-bit
 *   watermark key, a 64-bit context label Lambda(c) and a 32-bit position.
 * - `status` (nullable) is a device word the kernels OR flags into
 *   (PPS_FLAG_*); clear it before the call if you read it.
 *
 * The keyed source (this library's reading; the paper fixes only a keyed
 * pseudorandom function, Sec. 3.1 Eq. 1, and G(k, c), Alg. 3):
 *   word w(i, j) of token i, arrival j >= 1 = lane (i & 3) of
 *   Philox4x32-10(counter = (i >> 2, pos, ctx_lo, ctx_hi),
 *                 key = (key_lo ^ (j - 1) * 0x9E3779B9, key_hi)),
 *   u = (w + 1/2) 2^-32, E = -ln u ~ Exp(1) (first arrival, Thm A.1).
 *   Race key of token i at temperature T: s_i = ln E_i - logit_i / T
 *   (argmin s = argmin E/P, Alg. 2 and App. A.2); NaN logits never win.
 *   Ties in s go to the smaller token index.
 */
#ifndef PPS_H
#define PPS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* pps_stream_t; /* identical to cudaStream_t */

typedef enum {
    PPS_OK = 0,
    PPS_ERR_INVALID_ARG = 1, /* null pointer, size out of range, K > vocab, stride < vocab, T <= 0 ... */
    PPS_ERR_UNSUPPORTED = 2, /* dtype or mode not implemented                                        */
    PPS_ERR_WORKSPACE = 3,   /* workspace null or smaller than pps_workspace_size()                    */
    PPS_ERR_CUDA = 4,        /* a kernel launch or CUDA call failed                                    */
    PPS_ERR_SIZE = 5         /* problem larger than the fixed scratch of pps_draft_list_noalloc        */
} pps_status;

typedef enum { PPS_F32 = 0, PPS_BF16 = 1 } pps_dtype;

typedef enum {
    PPS_DRAFT_DISTINCT = 0, /* the K smallest first-arrival keys (K distinct tokens)                 */
    PPS_DRAFT_IID = 1       /* the K smallest multi-arrival scores (direct finite-support MPFR, App. B) */
} pps_draft_mode;

/* per-row identities, each an array of n_rows (device) */
typedef struct {
    const uint64_t* key;      /* watermark key k                         */
    const uint64_t* ctx_hash; /* context label Lambda(c)                 */
    const uint32_t* pos;      /* position of the context                 */
} pps_row_ids;

/* bits OR-ed into *status */
#define PPS_FLAG_GUARD 1u       /* fp32 streaming filter could not prove a row's candidate set complete */
#define PPS_FLAG_LOGIT_RANGE 2u /* |logit / T| too large for the fp32 filter's error bound (> 2^16)      */
#define PPS_FLAG_TREE 4u        /* a sequence's root row (seq_off[s]) lies outside the node rows: nothing emitted */
#define PPS_FLAG_TIMEOUT 8u     /* an LM-head kernel gave up waiting on its pipeline and returned early         */

#define PPS_MAX_K 32

/* Library version string and a text for a status code (host pointers, static). */
const char* pps_version(void);
const char* pps_status_string(pps_status s);

/* Rounds of the keyed source's Philox4x32 in this build of the library: 10
 * (libpps.so, Philox4x32-10 of Salmon et al., SC'11: every word, list, winner
 * and score of the other entry points follows it) or 7 (libpps_r7.so, built
 * with PPS_PHILOX_ROUNDS=7: the same counters and keys, three rounds fewer; a
 * different keyed source, so its outputs differ from libpps.so's).  The
 * paper's method needs a keyed pseudorandom function (Sec. 3.1); which
 * variant a deployment uses is fixed when it picks the library. */
int pps_philox_rounds(void);

/* Bytes of workspace pps_draft_list / pps_verify_tree need for n_rows rows and
 * n_seq sequences (n_seq = 0 for pps_draft_list).  The workspace holds
 * per-row partial candidate lists, arrival counters and the shared filter
 * bounds of rows cut between CTAs; it must be zeroed once
 * before its first use (pps_workspace_clear or cudaMemset) and is left zeroed
 * by every call that returns PPS_OK and runs to completion.  One workspace
 * must not be used by two calls that run concurrently. */
size_t pps_workspace_size(int64_t n_rows, int64_t vocab, int32_t K, int32_t n_seq);
pps_status pps_workspace_clear(void* ws, size_t ws_bytes, pps_stream_t stream);

/*
 * pps_draft_list -- the drafter's list at every context row (MPFR(Q(.|c),
 * Pi(c), nu(c)), Eq. 4; direct finite-support MPFR algorithm and the draft
 * side of the batched direct top-k algorithm, App. B; draft-tree step of
 * Alg. 4).
 *
 * q_logits     [n_rows, row_stride] draft logits (dtype), row r = context c_r
 * ids          identities of the n_rows contexts
 * temperature  T > 0, applied as logit / T
 * K            list stride and largest list length, 1 <= K <= min(32, vocab)
 * row_k        nullable [n_rows]: list length nu(c_r) of each row, 1..K
 *              (NULL = K for every row)
 * mode         PPS_DRAFT_DISTINCT or PPS_DRAFT_IID
 * out_tok      [n_rows, K] tokens of the k_r smallest first-arrival keys in
 *              ascending key order; -1 past k_r or past the row's usable tokens
 * out_key      nullable [n_rows, K] their keys s (fp32 estimate, natural log)
 * out_mult     [n_rows, K] DISTINCT: 1 per valid entry; IID: how many of the
 *              k_r samples carry the label out_tok[r, m]
 * out_ndistinct [n_rows] |D(c_r)|, the number of distinct draft tokens; they
 *              are out_tok[r, 0 .. out_ndistinct[r]-1] in both modes
 * out_samples  nullable [n_rows, K] the ordered samples (DISTINCT: = out_tok;
 *              IID: labels of the k_r smallest multi-arrival scores)
 * ws, ws_bytes workspace of pps_workspace_size(n_rows, vocab, K, 0) bytes
 */
pps_status pps_draft_list(const void* q_logits, pps_dtype dtype, int64_t n_rows, int64_t vocab, int64_t row_stride,
                          pps_row_ids ids, float temperature, int32_t K, const int32_t* row_k, pps_draft_mode mode,
                          int32_t* out_tok, float* out_key, int32_t* out_mult, int32_t* out_ndistinct,
                          int32_t* out_samples, uint32_t* status, void* ws, size_t ws_bytes, pps_stream_t stream);

/*
 * pps_verify_tree -- target race at every node of the draft trees, then the
 * walk along the realised target path with the watermark score of every
 * emitted token (batched-target evaluation and "follow the realised target
 * path" of the batched direct top-k algorithm, App. B; Alg. 4; score Eq. 2).
 *
 * p_logits     [n_nodes, row_stride] target logits, one row per tree node
 * ids          identities of the n_nodes contexts (the same labels the draft
 *              rows of those contexts used)
 * n_seq, gamma sequences and block length (1 <= gamma <= 64)
 * seq_off      [n_seq+1] sequence b owns nodes seq_off[b] .. seq_off[b+1]-1,
 *              its root is node seq_off[b] (non-decreasing, seq_off[0] = 0,
 *              seq_off[n_seq] = n_nodes)
 * node_draft_row [n_nodes] draft row of node c, -1 for a leaf
 * n_draft      number of draft rows
 * draft_tok, draft_ndistinct  pps_draft_list outputs for the draft rows
 *              ([n_draft, K], [n_draft]); D(c) = draft_tok[dr, 0..ndist-1]
 *              The walk treats a draft row outside [0, n_draft) as a leaf, a
 *              child outside [0, n_nodes) as not evaluated, and clamps ndist
 *              to K, so an inconsistent tree cannot make it read out of bounds;
 *              every sequence must own at least its root node, otherwise its
 *              outputs are not written.
 * K            stride of draft_tok and child_node
 * child_node   [n_draft, K] node reached from draft row dr by list slot m
 *              (the context c || draft_tok[dr, m]); -1 = not evaluated
 * out_winner   [n_nodes] y(c) = argmin_i s_i, -1 if no token is usable
 * out_word     [n_nodes] first-arrival word of y(c) (0 if none)
 * out_accept_len [n_seq] accepted steps (0..gamma)
 * out_n_emitted  [n_seq] emitted tokens (accept_len + 1, unless a winner was -1)
 * out_emitted  [n_seq, gamma+1] emitted tokens, -1 past the end
 * out_score    [n_seq, gamma+1] A = -ln(1 - u_y) of each emitted token, 0 past the end
 * out_score_sum [n_seq] sum of A (fp64)
 * ws, ws_bytes workspace of pps_workspace_size(n_nodes, vocab, 1, n_seq) bytes
 */
pps_status pps_verify_tree(const void* p_logits, pps_dtype dtype, int64_t n_nodes, int64_t vocab, int64_t row_stride,
                           pps_row_ids ids, float temperature, int32_t n_seq, int32_t gamma, const int32_t* seq_off,
                           const int32_t* node_draft_row, int64_t n_draft, const int32_t* draft_tok,
                           const int32_t* draft_ndistinct, int32_t K, const int32_t* child_node, int32_t* out_winner, uint32_t* out_word,
                           int32_t* out_accept_len, int32_t* out_n_emitted, int32_t* out_emitted, float* out_score,
                           double* out_score_sum, uint32_t* status, void* ws, size_t ws_bytes, pps_stream_t stream);

/*
 * Truncated calls -- pps_draft_list / pps_verify_tree with the logit
 * processing of the experiments (top-k = 50, top-p = 1 in Sec. 6) applied to
 * each row before the race; a truncated distribution has a support of at
 * most k tokens (Sec. 4.2).  Tokens outside the kept set S get P = 0
 * (E/P = +inf), so the race, lists, walk and scores are those of the
 * renormalised truncated distributions of P and Q.
 *
 * top_k        1 <= top_k <= PPS_MAX_TOP_K: S holds every token whose logit is
 *              >= the top_k-th largest usable logit (ties of it included;
 *              NaN and -inf logits never; all usable tokens if fewer than top_k)
 * top_p        0 < top_p <= 1: then, with probabilities softmax(logit / T) over
 *              the top-k set, whole groups of equal logits are removed from the
 *              bottom while the running mass, summed token by token in
 *              ascending logit order, is <= 1 - top_p; the largest group stays.
 *              1 = no top-p.
 * Every other argument, output and the workspace size are those of
 * pps_draft_list / pps_verify_tree.  PPS_ERR_INVALID_ARG for top_k or top_p
 * out of range.  A row whose top-k tie group does not fit the 64-entry list
 * is still exact: it is finished with a second pass over its logits.
 */
#define PPS_MAX_TOP_K 64

pps_status pps_draft_list_trunc(const void* q_logits, pps_dtype dtype, int64_t n_rows, int64_t vocab,
                                int64_t row_stride, pps_row_ids ids, float temperature, int32_t top_k, float top_p,
                                int32_t K, const int32_t* row_k, pps_draft_mode mode, int32_t* out_tok,
                                float* out_key, int32_t* out_mult, int32_t* out_ndistinct, int32_t* out_samples,
                                uint32_t* status, void* ws, size_t ws_bytes, pps_stream_t stream);

pps_status pps_verify_tree_trunc(const void* p_logits, pps_dtype dtype, int64_t n_nodes, int64_t vocab,
                                 int64_t row_stride, pps_row_ids ids, float temperature, int32_t top_k, float top_p,
                                 int32_t n_seq, int32_t gamma, const int32_t* seq_off, const int32_t* node_draft_row,
                                 int64_t n_draft, const int32_t* draft_tok, const int32_t* draft_ndistinct, int32_t K,
                                 const int32_t* child_node, int32_t* out_winner, uint32_t* out_word,
                                 int32_t* out_accept_len, int32_t* out_n_emitted, int32_t* out_emitted,
                                 float* out_score, double* out_score_sum, uint32_t* status, void* ws,
                                 size_t ws_bytes, pps_stream_t stream);

/*
 * pps_tree_expand -- one depth of the dynamic IID draft tree (Alg. 4 with
 * MPFR lists, Eq. 4): each present context c of depth d drew nu(c) i.i.d.
 * samples (pps_draft_list in PPS_DRAFT_IID mode with row_k = nu); every
 * distinct label u becomes a child c||u of depth d+1 that draws
 * nu(c||u) = mult(u) samples, so each sequence keeps K draft paths at every
 * depth and has at most K nodes per depth.  Child identity: the same key,
 * position + 1, label SplitMix64-output(label(c) ^ (u + 1) * 0x9E3779B97F4A7C15).
 *
 * Fixed-capacity layout (static; nothing else is reallocated per depth):
 *   nodes      N1 = 1 + K*gamma per sequence; node (b, d, i) =
 *              b*N1 + (d == 0 ? 0 : 1 + (d-1)*K + i); seq_off[b] = b*N1
 *   draft rows depth-major, n_seq*(1 + K*(gamma-1)) in all: depth d's rows
 *              start at D_d = n_seq*(d == 0 ? 0 : 1 + (d-1)*K), w_d = (d == 0 ?
 *              1 : K) per sequence, and node (b, d, i), d < gamma, owns draft
 *              row D_d + b*w_d + i (node_draft_row).  A depth's rows are the
 *              contiguous rows one pps_draft_list call takes.
 * Inputs (depth d's rows (b, i) = b*w_d + i, [n_seq*w_d]): draft_tok, draft_mult, draft_ndistinct
 * (pps_draft_list outputs, stride K), rows (their identities), row_k (nu; 0 =
 * an absent node, whose list is ignored).
 * Outputs: next_key, next_ctx, next_pos, next_k [n_seq*K]: identities and nu
 * of depth d+1's rows in child order (nu = 0 past the last child);
 * child_node [all draft rows, K]: the rows of depth d get their children's node
 * indices (-1 past ndistinct); node_key, node_ctx, node_pos [n_seq*N1]:
 * identities of depth d+1's nodes.  All device pointers.
 */
pps_status pps_tree_expand(int32_t n_seq, int32_t K, int32_t gamma, int32_t depth, const int32_t* draft_tok,
                           const int32_t* draft_mult, const int32_t* draft_ndistinct, pps_row_ids rows,
                           const int32_t* row_k, uint64_t* next_key, uint64_t* next_ctx, uint32_t* next_pos,
                           int32_t* next_k, int32_t* child_node, uint64_t* node_key, uint64_t* node_ctx,
                           uint32_t* node_pos, pps_stream_t stream);

/*
 * Non-identical proposals (App. A, the proposition on heterogeneous
 * proposals): B draft models Q_0..Q_{B-1} each propose one token per context
 * from one Poisson process on the augmented vocabulary V x [B].  Proposal b
 * is the race of Q_b over block b; the target is the race of P(i)/B over all
 * of V x [B], whose token Y is accepted iff it equals some proposal.
 *
 * The augmented source (this library's reading; the paper fixes only that
 * the points of V x [B] carry one common Poisson process): the B first
 * arrivals of token i are generated by competing exponentials,
 *   E_(i,b) = E'_i / B                    for b = J_i,
 *   E_(i,b) = E'_i / B + F_(i,b)          otherwise,
 * E'_i = -ln u of word w(i, 1) under the row's key (the plain source),
 * J_i = floor(B w' / 2^32), w' = token i's word under key ^ 0x3C6EF372FE94F82B,
 * F_(i,b) = -ln u of token i's word under key ^ (b + 1) * 0xBB67AE8584CAA73B
 * (the least of B iid Exp(1) is Exp(B), in a uniform block independent of
 * its value; the rest exceed it by iid Exp(1)).  Consequences: the target's Y
 * is exactly the plain race winner on P (pps_verify_tree), its watermark word
 * and the detector (pps_wm_score / pps_wm_detect) are unchanged, and J = J_Y
 * (pps_hetero_block).
 */
#define PPS_MAX_BLOCKS 32

/*
 * pps_draft_hetero -- proposal rows: row r is proposal b = row_block[r] at
 * its context, X = argmin_i ln E_(i,b) - logit_i / T (ties to the smaller
 * token).  Arguments as pps_draft_list with K = 1, plus:
 * row_block    [n_rows] proposal index of each row, 0 <= b < n_blocks (other
 *              values are read as block indices of the same source; no memory
 *              is indexed by them)
 * n_blocks     B, 1 <= B <= PPS_MAX_BLOCKS (B = 1 is the plain race)
 * out_tok      [n_rows] X, -1 if no token is usable
 * out_key      nullable [n_rows] its key s = ln E_(X,b) - logit_X / T (fp32)
 * ws, ws_bytes workspace of pps_workspace_size(n_rows, vocab, 1, 0) bytes
 */
pps_status pps_draft_hetero(const void* q_logits, pps_dtype dtype, int64_t n_rows, int64_t vocab, int64_t row_stride,
                            pps_row_ids ids, float temperature, const int32_t* row_block, int32_t n_blocks,
                            int32_t* out_tok, float* out_key, uint32_t* status, void* ws, size_t ws_bytes,
                            pps_stream_t stream);

/*
 * pps_draft_hetero_trunc -- pps_draft_hetero with the logit processing of the
 * truncated calls (top_k, top_p as pps_draft_list_trunc) applied to each
 * proposal row before its race: proposal b races its truncated Q_b over
 * block b.  PPS_ERR_INVALID_ARG for top_k or top_p out of range.
 */
pps_status pps_draft_hetero_trunc(const void* q_logits, pps_dtype dtype, int64_t n_rows, int64_t vocab,
                                  int64_t row_stride, pps_row_ids ids, float temperature, int32_t top_k, float top_p,
                                  const int32_t* row_block, int32_t n_blocks, int32_t* out_tok, float* out_key,
                                  uint32_t* status, void* ws, size_t ws_bytes, pps_stream_t stream);

/*
 * pps_hetero_expand -- one depth of the draft tree of B proposals, each
 * drafting a chain of gamma tokens (each row drafted by pps_draft_hetero);
 * chains that agree share nodes, so node c's draft list D(c) is the set of
 * distinct tokens its proposals drew, and pps_verify_tree walks the tree with
 * K = B.  A proposal at node o of depth d that drew x moves to the child
 * (d+1, f), f = the first proposal at o that drew x.  Child identity: the same
 * key, position + 1, label SplitMix64-output(label(c) ^ (x + 1) *
 * 0x9E3779B97F4A7C15) (as pps_tree_expand).
 *
 * Fixed-capacity layout (K = B in pps_tree_expand's formulas):
 *   nodes        N1 = 1 + B*gamma per sequence; node (s, d, o) =
 *                s*N1 + (d == 0 ? 0 : 1 + (d-1)*B + o); seq_off[s] = s*N1;
 *                node (s, d+1, b) is used iff proposal b is the first to reach it
 *   node lists   depth-major, n_seq*(1 + B*(gamma-1)) rows of stride B: depth
 *                d's rows start at L_d = n_seq*(d == 0 ? 0 : 1 + (d-1)*B),
 *                w_d = (d == 0 ? 1 : B) per sequence, node (s, d, o) owns list
 *                row L_d + s*w_d + o (its node_draft_row)
 *   proposal rows depth-major, n_seq*B per depth: row (s, b) = s*B + b
 * Inputs (depth d's proposal rows): draft_tok [n_seq*B] (pps_draft_hetero
 * outputs), rows (their identities), row_owner [n_seq*B]: the node (s, d, o)
 * of each row as o (0 at depth 0), -1 = proposal stopped (it drew nothing at
 * an earlier depth).  A row with draft_tok < 0 stops its proposal.
 * Outputs: list_tok, child_node [n_lists, B] and list_ndistinct [n_lists]:
 * depth d's lists (tokens in proposal order, -1 past ndistinct; every list
 * row of the depth is written, 0 entries for unused nodes); node_key,
 * node_ctx, node_pos [n_seq*N1]: depth d+1's nodes (zeros for unused ones);
 * next_key, next_ctx, next_pos, next_owner [n_seq*B]: depth d+1's proposal
 * rows (only when depth + 1 < gamma; nullable otherwise).  All device pointers.
 */
pps_status pps_hetero_expand(int32_t n_seq, int32_t n_blocks, int32_t gamma, int32_t depth, const int32_t* draft_tok,
                             pps_row_ids rows, const int32_t* row_owner, uint64_t* next_key, uint64_t* next_ctx,
                             uint32_t* next_pos, int32_t* next_owner, int32_t* list_tok, int32_t* list_ndistinct,
                             int32_t* child_node, uint64_t* node_key, uint64_t* node_ctx, uint32_t* node_pos,
                             pps_stream_t stream);

/*
 * pps_hetero_block -- the block J = J_Y of the target's augmented point
 * (Y, J) for n tokens Y (e.g. pps_verify_tree winners) under their contexts'
 * identities; -1 where Y < 0.  1 <= n_blocks <= PPS_MAX_BLOCKS.
 */
pps_status pps_hetero_block(const int32_t* tokens, pps_row_ids ids, int64_t n, int32_t n_blocks, int32_t* out_block,
                            pps_stream_t stream);

/*
 * pps_wm_score -- detector pass (detector algorithm of App. E; Eq. 2):
 * regenerate the first-arrival word of every observed token under its
 * context's identity and score it, A_t = -ln(1 - u_t).
 *
 * tokens       [n] observed tokens (0 <= token < 2^34)
 * ids          [n] identity of the context each token was emitted in
 * n_seg, seg_off  nullable seg_off [n_seg+1]: segment g = tokens
 *              seg_off[g] .. seg_off[g+1]-1 (non-decreasing, seg_off[0] = 0,
 *              seg_off[n_seg] = n); NULL = one segment of all n tokens
 * out_score    nullable [n] A_t (fp32; relative error below 2.2e-6, absolute below 2e-7)
 * out_sum      nullable [n_seg] (or [1]) S_A per segment (fp64; the fp32 scores summed with
 *              fp32 warp reductions into a compensated float-float running sum); zeroed by
 *              the call
 */
pps_status pps_wm_score(const int32_t* tokens, pps_row_ids ids, int64_t n, int32_t n_seg, const int64_t* seg_off,
                        float* out_score, double* out_sum, pps_stream_t stream);

/*
 * pps_wm_detect -- the detector pass with a choice of per-token score of the
 * same pivot r = u (App. D) and per-segment log p-values (App. D.2; detector
 * algorithm, App. E).  Arguments as pps_wm_score, plus:
 *
 * kind         PPS_SCORE_AARONSON  -ln(1 - r)                    (param unused)
 *              PPS_SCORE_U         r, the U-score                (param unused)
 *              PPS_SCORE_LI        Li et al.'s optimal Gumbel score
 *                                  ln(k r^(D/(1-D)) + [q > 0] r^((1-q)/q)),
 *                                  k = floor(1/(1-D)), q = 1 - k(1-D); param D in (0, 1)
 *              PPS_SCORE_POWER_LAW Lattimore's truncated power law
 *                                  min(e^(-1/2), (1-r)^(-1/2)) - (2 - e^(1/2)); param e in (0, 1]
 * out_score    nullable [n] per-token scores (fp32)
 * out_sum      [n_seg] (or [1]) per-segment sums (fp64); zeroed by the call;
 *              nullable only when out_logp is NULL
 * out_logp     nullable [n_seg] (or [1]) natural log of the segment's null
 *              p-value, M = its token count: AARONSON ln P(Gamma(M,1) >= S)
 *              (to ~1e-6 absolute); U the Chernoff bound (its minimiser in
 *              fp32; the bound at it in fp64)
 *              inf_l M ln((e^l - 1)/l) - l S (0 for S <= M/2); NaN for the
 *              other kinds (the paper gives them no null law); 0 for M = 0.
 * PPS_ERR_INVALID_ARG for param out of range, PPS_ERR_UNSUPPORTED for kind.
 */
typedef enum {
    PPS_SCORE_AARONSON = 0,
    PPS_SCORE_U = 1,
    PPS_SCORE_LI = 2,
    PPS_SCORE_POWER_LAW = 3
} pps_score_kind;

pps_status pps_wm_detect(const int32_t* tokens, pps_row_ids ids, int64_t n, int32_t n_seg, const int64_t* seg_off,
                         pps_score_kind kind, double param, float* out_score, double* out_sum, double* out_logp,
                         pps_stream_t stream);

/*
 * LM head with the race fused into it (App. B: the batched-target algorithm
 * evaluates the target model once for every context of a draft block; the
 * race of Alg. 2 is then the only consumer of those logits).
 *
 *   logits[r, i] = sum_j hidden[r, j] * weight[i, j]
 *
 * hidden   [n_rows, d] bf16, row stride ld_hidden elements: the last hidden
 *          state of each context (node row or draft row)
 * weight   [vocab, d] bf16, row stride ld_weight elements: the LM-head matrix,
 *          one row per token
 * The product is formed on the tensor cores (tcgen05.mma, bf16 operands, fp32
 * accumulation) in 128 x 256 tiles with a fixed reduction order; the fp32
 * accumulators are the logits.  Both bases must be 16-byte aligned, both row
 * strides multiples of 8 elements (16 bytes), ld >= d; PPS_ERR_INVALID_ARG
 * otherwise.
 *
 * pps_lmhead_logits writes those logits to out_logits [n_rows, ld_out] fp32
 * (ld_out >= vocab): the unfused path, whose output the streaming entry points
 * (pps_draft_list, pps_verify_tree with PPS_F32) take.
 *
 * pps_lmhead_draft_list and pps_lmhead_verify_tree compute the same outputs
 * as pps_draft_list / pps_verify_tree would on those fp32 logits, bit for bit
 * (tokens, words, multiplicities, accept lengths, scores), without writing the
 * logits anywhere: the race runs on each accumulator tile in the GEMM's
 * epilogue, and a second small kernel merges each row's partial lists and
 * finishes the row (near-tie re-keying, IID epilogue, tree walk).  Draft lists
 * are limited to K <= PPS_LMHEAD_MAX_K.  A row whose kept candidates cannot
 * prove its list complete (more than one near tie at the k-th key) raises
 * PPS_FLAG_GUARD; PPS_FLAG_TIMEOUT reports a pipeline that gave up waiting
 * (outputs undefined).  The workspace holds the partial lists and the
 * sequence tickets: pps_lmhead_workspace_size bytes, zeroed once before first
 * use (pps_workspace_clear); the calls leave it ready for the next call.
 */
#define PPS_LMHEAD_MAX_K 8
size_t pps_lmhead_workspace_size(int64_t n_rows, int32_t n_seq);
pps_status pps_lmhead_logits(const void* hidden, int64_t ld_hidden, const void* weight, int64_t ld_weight,
                             int64_t n_rows, int64_t vocab, int64_t d, float* out_logits, int64_t ld_out,
                             pps_stream_t stream);
pps_status pps_lmhead_draft_list(const void* hidden, int64_t ld_hidden, const void* weight, int64_t ld_weight,
                                 int64_t n_rows, int64_t vocab, int64_t d, pps_row_ids ids, float temperature,
                                 int32_t K, const int32_t* row_k, pps_draft_mode mode, int32_t* out_tok,
                                 float* out_key, int32_t* out_mult, int32_t* out_ndistinct, int32_t* out_samples,
                                 uint32_t* status, void* ws, size_t ws_bytes, pps_stream_t stream);
pps_status pps_lmhead_verify_tree(const void* hidden, int64_t ld_hidden, const void* weight, int64_t ld_weight,
                                  int64_t n_nodes, int64_t vocab, int64_t d, pps_row_ids ids, float temperature,
                                  int32_t n_seq, int32_t gamma, const int32_t* seq_off, const int32_t* node_draft_row,
                                  int64_t n_draft, const int32_t* draft_tok, const int32_t* draft_ndistinct,
                                  int32_t K, const int32_t* child_node, int32_t* out_winner, uint32_t* out_word,
                                  int32_t* out_accept_len, int32_t* out_n_emitted, int32_t* out_emitted,
                                  float* out_score, double* out_score_sum, uint32_t* status, void* ws,
                                  size_t ws_bytes, pps_stream_t stream);

/*
 * pps_draft_list_noalloc -- pps_draft_list for callers that must not
 * allocate device memory per call and cannot hand the library a workspace:
 * code running under an allocator that forbids new allocations once serving
 * has started, plugin or callback hooks of an inference engine that receive
 * only their input and output buffers, or deployments that must size every
 * device buffer up front.  The paper has no counterpart; this is a packaging
 * variant of the draft-list entry point, with the same arguments minus the
 * workspace and the same outputs.
 *
 * Its scratch (per-row partial lists and arrival counters) is one file-scope
 * device array of PPS_NOALLOC_SCRATCH_BYTES (about 1.8 MB) that every GPU
 * which loads libpps holds until the process exits.  It serves at most
 * PPS_NOALLOC_MAX_ROWS rows per call (larger n_rows returns PPS_ERR_SIZE)
 * and caps the kernel grid at PPS_NOALLOC_MAX_WARPS warps.  The first call
 * on a device looks the array's device address up (a CUDA runtime query, no
 * allocation); make that first call before any stream capture.  Each call
 * clears the counters it uses with an asynchronous memset on `stream` and
 * allocates nothing.  All calls share the one array and it keeps the last
 * call's contents: calls whose executions overlap on the GPU (on different
 * streams, or from different threads without ordering) race on it, so the
 * caller must serialise them.
 */
#define PPS_NOALLOC_MAX_ROWS 4096
#define PPS_NOALLOC_MAX_WARPS 2432
/* bytes of the array: a 272-byte partial list per (row + warp) slot, then two
 * 32-bit counters per row: 272 * (4096 + 2432) + 8 * 4096 */
#define PPS_NOALLOC_SCRATCH_BYTES 1808384
pps_status pps_draft_list_noalloc(const void* q_logits, pps_dtype dtype, int64_t n_rows, int64_t vocab,
                                  int64_t row_stride, pps_row_ids ids, float temperature, int32_t K,
                                  const int32_t* row_k, pps_draft_mode mode, int32_t* out_tok, float* out_key,
                                  int32_t* out_mult, int32_t* out_ndistinct, int32_t* out_samples, uint32_t* status,
                                  pps_stream_t stream);

/* Raw words w(i, arrival) for i < vocab of n_rows rows -> out [n_rows, vocab]
 * (bit-exact check of the keyed source). */
pps_status pps_philox_words(pps_row_ids ids, int64_t n_rows, int64_t vocab, int32_t arrival, uint32_t* out,
                            pps_stream_t stream);

/* Self-test of the fp32 key transform used by the streaming filter: over
 * every 32-bit word w in [w_begin, w_end) it compares the fp32 value of
 * log2(-log2 u(w)) with an fp64 evaluation and writes the largest absolute
 * difference to out_max_err[0] (device float, must hold 0 before the call). */
pps_status pps_selftest_key_error(uint64_t w_begin, uint64_t w_end, float* out_max_err, pps_stream_t stream);

/* Self-test of the fp32 logarithm inside the block key of pps_draft_hetero:
 * over every fp32 x in [x_lo, x_hi) (0 < x_lo <= x_hi, finite) it compares
 * lg2.approx(x) with an fp64 log2 and writes the largest absolute difference
 * to out_max_err[0] (device float, must hold 0 before the call).  The block
 * key's error bound assumes at most 2^-17 over [2^-40, 2^7). */
pps_status pps_selftest_lg2_error(float x_lo, float x_hi, float* out_max_err, pps_stream_t stream);

/* Throughput self-test of the keyed source alone: generates n_blocks Philox
 * blocks (4 words each) with the streaming kernels' row-specialised
 * generator, in a grid of out_len / 256 CTAs of 256 threads, and writes one
 * folded word per thread to out [out_len] (device, out_len >= 256).  Timing
 * it gives the multiply-bound ceiling of the race kernels. */
pps_status pps_selftest_philox_rate(uint64_t n_blocks, uint32_t* out, int32_t out_len, pps_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* PPS_H */
