/*
 * pps_oracle.c -- plain, slow, double-precision CPU oracle for the keyed
 * Poisson-race (exponential race) multi-draft speculative sampler of
 * "Watermarkable Multi-Draft Speculative Sampling via Poisson Processes".
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this library.  It shares
 * no code, header, table or constant generator with the CUDA path; it is an
 * independent restatement of the paper's definitions, written for a reader to
 * check by eye, not for speed.  Rows are independent, so an OpenMP loop over
 * rows is the only concession to run time; it changes no arithmetic.
 *
 * What each function follows:
 *   orc_philox4x32_10  Philox4x32-10 counter-based generator (Salmon, Moraes,
 *                      Dror, Shaw, "Parallel random numbers: as easy as 1, 2, 3",
 *                      SC'11): 10 rounds of the 4x32 Philox S-box with the
 *                      published multipliers and Weyl key increments.  The
 *                      paper only asks for a keyed pseudorandom function
 *                      F_{ctx,k} (Sec. 3.1, Eq. 1) / keyed source G(k,c)
 *                      (Alg. 3); Philox is the reading taken here.
 *   orc_philox4x32     the same with R rounds (Philox4x32-R); the keyed source
 *                      uses R = orc_set_philox_rounds() (10, or 7 for the
 *                      cheaper variant a library build can select).  Pinned
 *                      through the 10-round known answers: R rounds followed by
 *                      10 - R rounds under the key advanced by R Weyl steps are
 *                      the 10-round function.
 *   orc_word           the keyed source Pi_k(c): counter (token>>2, pos,
 *                      ctx_lo, ctx_hi), key (key_lo ^ (j-1)*0x9E3779B9, key_hi)
 *                      for arrival j, output lane token&3.
 *   orc_exp1           E = -ln u with u = (w + 1/2) 2^-32 (first arrival time
 *                      scaled to Exp(1), Thm A.1 Eq. "E_z = q_z S_z").
 *   orc_race_key       s = ln E - l/T, the log of E/p up to a row constant
 *                      (exponential race, Alg. 2; Gumbel-max equivalence,
 *                      App. A.2).
 *   orc_target_rows    y(c) = argmin_i E_i / P(i) (EFR, Thm A.1; target side of
 *                      the batched direct top-k algorithm, App. B).
 *   orc_draft_rows     DISTINCT: the K smallest E_i/Q(i) (first arrivals);
 *                      IID: the K smallest multi-arrival scores
 *                      G_{u,j}/Q(u), G_{u,j} = sum_{m<=j} E_{u,m}, j = 1..K,
 *                      over every token u with Q(u) > 0 (direct finite-support
 *                      MPFR algorithm, App. B, Thm "exactness of direct
 *                      finite-support MPFR").
 *   orc_lmhead_logits  logits = hidden . weight^T in fp64 (the LM head whose
 *                      output the race consumes; App. B cost remark).
 *   orc_walk           follow the realised target path through the context
 *                      tree, accept while y(c*) is in D(c*), bonus token after
 *                      gamma acceptances (Alg. 4; batched algorithm, App. B).
 *   orc_wm_score       A_t = -ln(1 - r_t(w_t)) with pivot r_t = u of the
 *                      emitted token (Eq. 2; App. D.1 "Gumbel watermark";
 *                      detector algorithm, App. E).
 *   orc_score_kind     per-token detection scores of the same pivot r = u
 *                      (App. D): Aaronson A = -ln(1 - r); the U-score r;
 *                      Li et al.'s optimal Gumbel score h*_{gum,Delta}(r) =
 *                      ln(k r^(Delta/(1-Delta)) + [q > 0] r^((1-q)/q)),
 *                      k = floor(1/(1-Delta)), q = 1 - k(1-Delta); Lattimore's
 *                      truncated power law min(eps^-1/2, (1-r)^-1/2) - (2 - sqrt eps).
 *   orc_gamma_tail_logp  ln P(Gamma(M,1) >= S), the exact null p-value of S_A
 *                      (App. D.2; detector algorithm, App. E), for integer M as
 *                      the Poisson sum P(Poisson(S) <= M - 1).
 *   orc_chernoff_u_logp  the Chernoff bound on the U-score tail,
 *                      inf over lambda >= 0 of M ln((e^lambda - 1)/lambda) - lambda S
 *                      (App. D.2), by golden-section search on the convex exponent.
 *   orc_tree_expand    one depth of the dynamic IID draft tree (Alg. 4 with
 *                      MPFR lists, Eq. 4): every distinct label u of a
 *                      context's k_r i.i.d. draft samples becomes a child
 *                      c||u that draws nu(c||u) = its multiplicity samples at
 *                      the next depth, so the draft paths of a sequence stay
 *                      K at every depth.  Child context label: SplitMix64's
 *                      output function of label(c) ^ ((u + 1) * 0x9E3779B97F4A7C15)
 *                      (a reading: the paper leaves the labeler open),
 *                      position + 1, same key.
 *   orc_hetero_rows    non-identical proposals Q_0..Q_{B-1} (App. A, the
 *                      proposition on heterogeneous proposals): one Poisson
 *                      process on the augmented vocabulary V x [B]; proposal b
 *                      races Q_b over block b, the target races P(i)/B over all
 *                      (i, b); Y is accepted iff it equals some X^(b).
 *   orc_block_draft_rows  proposal b's race alone, per row (tree drafting).
 *   orc_truncate_rows  the logit processing of the experiments (Sec. 6 setup:
 *                      top-k = 50, top-p = 1; truncation leaves a support of at
 *                      most k tokens, Sec. 4.2): tokens outside the top-k /
 *                      top-p set get logit -inf, i.e. P = 0 and E/P = +inf, so
 *                      the race over the masked row is the race of the
 *                      truncated distribution.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------ */
/* Philox4x32-10                                                       */
/* ------------------------------------------------------------------ */

/* multipliers and Weyl key increments published for Philox4x32 */
#define ORC_PHILOX_M0 0xD2511F53u
#define ORC_PHILOX_M1 0xCD9E8D57u
#define ORC_PHILOX_W0 0x9E3779B9u
#define ORC_PHILOX_W1 0xBB67AE85u

/* Philox4x32 with `rounds` rounds (the same round function and key schedule;
 * Philox4x32-R of Salmon et al. for R = rounds). */
void orc_philox4x32(const uint32_t ctr_in[4], const uint32_t key_in[2], int rounds, uint32_t out[4])
{
    uint32_t x0 = ctr_in[0], x1 = ctr_in[1], x2 = ctr_in[2], x3 = ctr_in[3];
    uint32_t k0 = key_in[0], k1 = key_in[1];
    for (int round = 0; round < rounds; ++round) {
        if (round > 0) { /* key schedule: bump before every round but the first */
            k0 += ORC_PHILOX_W0;
            k1 += ORC_PHILOX_W1;
        }
        uint64_t p0 = (uint64_t)ORC_PHILOX_M0 * (uint64_t)x0;
        uint64_t p1 = (uint64_t)ORC_PHILOX_M1 * (uint64_t)x2;
        uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        uint32_t y0 = hi1 ^ x1 ^ k0;
        uint32_t y1 = lo1;
        uint32_t y2 = hi0 ^ x3 ^ k1;
        uint32_t y3 = lo0;
        x0 = y0; x1 = y1; x2 = y2; x3 = y3;
    }
    out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

void orc_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2], uint32_t out[4])
{
    orc_philox4x32(ctr_in, key_in, 10, out);
}

/* Rounds of the keyed source's Philox: 10 (the published default), or the
 * cheaper variant a library build selects (7).  Process-wide; set it before
 * any oracle computation.  r <= 0 only queries.  Returns the setting. */
static int orc_rounds = 10;
int orc_set_philox_rounds(int r)
{
    if (r > 0 && r <= 16) orc_rounds = r;
    return orc_rounds;
}

/* Keyed source: the 32-bit word of token `token`, arrival j >= 1, at the
 * context labelled (ctx, pos) under watermark key `key`. */
uint32_t orc_word(uint64_t key, uint64_t ctx, uint32_t pos, int64_t token, int32_t arrival)
{
    uint32_t ctr[4], k[2], out[4];
    ctr[0] = (uint32_t)((uint64_t)token >> 2);
    ctr[1] = pos;
    ctr[2] = (uint32_t)(ctx & 0xFFFFFFFFull);
    ctr[3] = (uint32_t)(ctx >> 32);
    uint32_t tweak = (uint32_t)(arrival - 1) * ORC_PHILOX_W0; /* 0 for the first arrival */
    k[0] = (uint32_t)(key & 0xFFFFFFFFull) ^ tweak;
    k[1] = (uint32_t)(key >> 32);
    orc_philox4x32(ctr, k, orc_rounds, out);
    return out[token & 3];
}

/* ------------------------------------------------------------------ */
/* uniform, exponential, race key, score                               */
/* ------------------------------------------------------------------ */

/* u = (w + 1/2) 2^-32, never 0 or 1, exact in double */
double orc_uniform(uint32_t w) { return ((double)w + 0.5) * 0x1p-32; }

/* 1 - u = (~w + 1/2) 2^-32, exact in double */
static double orc_one_minus_uniform(uint32_t w) { return ((double)(uint32_t)~w + 0.5) * 0x1p-32; }

/* E = -ln u ~ Exp(1).  For u > 1/2 the same value is written through
 * v = 1 - u so that small E keeps its relative precision. */
double orc_exp1(uint32_t w)
{
    if (w < 0x80000000u) return -log(orc_uniform(w));
    return -log1p(-orc_one_minus_uniform(w));
}

/* Aaronson per-token score A = -ln(1 - u) (Eq. 2). */
double orc_score_word(uint32_t w)
{
    if (w < 0x80000000u) return -log1p(-orc_uniform(w));
    return -log(orc_one_minus_uniform(w));
}

/* race key s = ln E - l/T.  A token with P = 0 (logit -inf) or an unusable
 * logit (NaN) never wins: key +inf.  A logit of +inf gives -inf. */
double orc_race_key(uint32_t w, double logit, double T)
{
    if (isnan(logit)) return INFINITY;
    return log(orc_exp1(w)) - logit / T;
}

/* (key, index) lexicographic order: ties go to the smaller token index */
static int orc_before(double ka, int64_t ia, double kb, int64_t ib)
{
    if (ka < kb) return 1;
    if (ka > kb) return 0;
    return ia < ib;
}

/* ------------------------------------------------------------------ */
/* target winner per row                                               */
/* ------------------------------------------------------------------ */

/* winner[r] = argmin_i s_i (or -1 if every key is +inf); word[r] its first-
 * arrival word; key[r] its key; margin[r] = s_(2) - s_(1) (+inf if < 2). */
void orc_target_rows(const float* logits, int64_t n_rows, int64_t V, int64_t stride, double T,
                     const uint64_t* key, const uint64_t* ctx, const uint32_t* pos,
                     int32_t* winner, uint32_t* word, double* key_out, double* margin)
{
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < n_rows; ++r) {
        const float* l = logits + r * stride;
        double best = INFINITY, second = INFINITY;
        int64_t bi = -1, si = -1;
        for (int64_t i = 0; i < V; ++i) {
            uint32_t w = orc_word(key[r], ctx[r], pos[r], i, 1);
            double s = orc_race_key(w, (double)l[i], T);
            if (s == INFINITY) continue;
            if (bi < 0 || orc_before(s, i, best, bi)) {
                second = best; si = bi;
                best = s; bi = i;
            } else if (si < 0 || orc_before(s, i, second, si)) {
                second = s; si = i;
            }
        }
        winner[r] = (int32_t)bi;
        if (word) word[r] = bi >= 0 ? orc_word(key[r], ctx[r], pos[r], bi, 1) : 0u;
        if (key_out) key_out[r] = best;
        if (margin) margin[r] = (bi >= 0 && si >= 0) ? second - best : INFINITY;
    }
}

/* ------------------------------------------------------------------ */
/* draft lists                                                         */
/* ------------------------------------------------------------------ */

typedef struct { double s; int64_t i; int32_t j; } orc_cand;

static int orc_cand_cmp(const void* a, const void* b)
{
    const orc_cand* x = (const orc_cand*)a;
    const orc_cand* y = (const orc_cand*)b;
    if (x->s < y->s) return -1;
    if (x->s > y->s) return 1;
    if (x->i != y->i) return x->i < y->i ? -1 : 1;
    if (x->j != y->j) return x->j < y->j ? -1 : 1;
    return 0;
}

/* mode 0 = DISTINCT, 1 = IID.
 * Per row r with list length k_r = row_k ? row_k[r] : K:
 *   tok[r*K + m]   m-th smallest first-arrival key (ascending, ties by index),
 *                  -1 past the end of the usable tokens or past k_r;
 *   keys[r*K + m]  its key (+inf when tok = -1);
 *   mult[r*K + m]  DISTINCT: 1 for a valid entry; IID: how many of the k_r
 *                  multi-arrival samples carry label tok[m];
 *   ndist[r]       number of distinct draft tokens |D(c)|;
 *   labels[r*K+m]  (nullable) the ordered samples: DISTINCT = tok, IID = the
 *                  labels U_(1..k_r) of the k_r smallest scores;
 *   min_gap[r]     (nullable) smallest gap between consecutive first-arrival
 *                  keys s_(m+1) - s_(m), m = 1..k_r (flip accounting).
 */
void orc_draft_rows(const float* logits, int64_t n_rows, int64_t V, int64_t stride, double T,
                    const uint64_t* key, const uint64_t* ctx, const uint32_t* pos,
                    int32_t K, const int32_t* row_k, int32_t mode,
                    int32_t* tok, double* keys, int32_t* mult, int32_t* ndist,
                    int32_t* labels, double* min_gap)
{
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < n_rows; ++r) {
        const float* l = logits + r * stride;
        int32_t kr = row_k ? row_k[r] : K;
        orc_cand* first = (orc_cand*)malloc(sizeof(orc_cand) * (size_t)V);
        int64_t n_use = 0;
        for (int64_t i = 0; i < V; ++i) {
            uint32_t w = orc_word(key[r], ctx[r], pos[r], i, 1);
            double s = orc_race_key(w, (double)l[i], T);
            if (s == INFINITY) continue;
            first[n_use].s = s; first[n_use].i = i; first[n_use].j = 1;
            ++n_use;
        }
        qsort(first, (size_t)n_use, sizeof(orc_cand), orc_cand_cmp);
        for (int32_t m = 0; m < K; ++m) {
            int ok = m < kr && m < n_use;
            tok[r * K + m] = ok ? (int32_t)first[m].i : -1;
            if (keys) keys[r * K + m] = ok ? first[m].s : INFINITY;
            mult[r * K + m] = 0;
            if (labels) labels[r * K + m] = -1;
        }
        if (min_gap) {
            double g = INFINITY;
            for (int32_t m = 0; m < kr && m + 1 < n_use; ++m) {
                double d = first[m + 1].s - first[m].s;
                if (d < g) g = d;
            }
            min_gap[r] = g;
        }
        int32_t nvalid = kr < n_use ? kr : (int32_t)n_use;
        if (mode == 0) {
            for (int32_t m = 0; m < nvalid; ++m) {
                mult[r * K + m] = 1;
                if (labels) labels[r * K + m] = (int32_t)first[m].i;
            }
            ndist[r] = nvalid;
        } else {
            /* every usable token u contributes arrivals j = 1..k_r with score
             * ln(G_{u,j}) - l_u/T; keep the k_r smallest */
            int64_t nc = n_use * (int64_t)kr;
            orc_cand* all = (orc_cand*)malloc(sizeof(orc_cand) * (size_t)(nc > 0 ? nc : 1));
            int64_t c = 0;
            for (int64_t i = 0; i < V; ++i) {
                double li = (double)l[i];
                if (isnan(li) || li == -INFINITY) continue;
                double G = 0.0;
                for (int32_t j = 1; j <= kr; ++j) {
                    G += orc_exp1(orc_word(key[r], ctx[r], pos[r], i, j));
                    all[c].s = log(G) - li / T;
                    all[c].i = i; all[c].j = j;
                    ++c;
                }
            }
            qsort(all, (size_t)c, sizeof(orc_cand), orc_cand_cmp);
            int32_t ns = kr < c ? kr : (int32_t)c;
            for (int32_t m = 0; m < ns; ++m) {
                if (labels) labels[r * K + m] = (int32_t)all[m].i;
                for (int32_t q = 0; q < nvalid; ++q)
                    if (tok[r * K + q] == (int32_t)all[m].i) { mult[r * K + q] += 1; break; }
            }
            int32_t nd = 0;
            for (int32_t q = 0; q < nvalid; ++q) nd += mult[r * K + q] > 0;
            ndist[r] = nd;
            free(all);
        }
        free(first);
    }
}

/* ------------------------------------------------------------------ */
/* tree walk and per-token score                                       */
/* ------------------------------------------------------------------ */

/* Sequence b owns nodes [seq_off[b], seq_off[b+1]); its root is seq_off[b].
 * Node c has draft row dr = node_draft_row[c] (-1 for a leaf); D(c) is
 * draft_tok[dr*K + m] for m < draft_ndist[dr], and child_node[dr*K + m] is
 * the node reached by that token (-1 if the caller evaluated none).
 * Outputs per sequence: accept_len (accepted steps, 0..gamma), n_emitted,
 * emitted[b*(gamma+1) + t], score[...] (A of each emitted token, 0 past the
 * end, emitted = -1 past the end), score_sum[b] (sum of A). */
void orc_walk(int32_t n_seq, int32_t gamma, const int32_t* seq_off, const int32_t* node_draft_row,
              const int32_t* draft_tok, const int32_t* draft_ndist, int32_t K, const int32_t* child_node,
              const int32_t* winner, const uint32_t* word,
              int32_t* accept_len, int32_t* n_emitted, int32_t* emitted, double* score, double* score_sum)
{
    for (int32_t b = 0; b < n_seq; ++b) {
        int32_t W = gamma + 1;
        for (int32_t t = 0; t < W; ++t) { emitted[b * W + t] = -1; score[b * W + t] = 0.0; }
        int32_t c = seq_off[b], acc = 0, ne = 0;
        double S = 0.0;
        int stopped = 0;
        for (int32_t s = 0; s < gamma; ++s) {
            int32_t y = winner[c];
            if (y < 0) { stopped = 1; break; }
            double A = orc_score_word(word[c]);
            emitted[b * W + ne] = y; score[b * W + ne] = A; S += A; ++ne;
            int32_t dr = node_draft_row[c], found = -1;
            if (dr >= 0)
                for (int32_t m = 0; m < draft_ndist[dr]; ++m)
                    if (draft_tok[dr * K + m] == y) { found = m; break; }
            if (found < 0) { stopped = 1; break; }
            int32_t nxt = child_node[dr * K + found];
            if (nxt < 0) { stopped = 1; break; }
            c = nxt; ++acc;
        }
        if (!stopped && winner[c] >= 0) {
            double A = orc_score_word(word[c]);
            emitted[b * W + ne] = winner[c]; score[b * W + ne] = A; S += A; ++ne;
        }
        accept_len[b] = acc; n_emitted[b] = ne; score_sum[b] = S;
    }
}

/* Detector pass: per token A_t from the regenerated first-arrival word, and
 * per segment sums (seg_off[n_seg+1]; nullable -> one segment). */
void orc_wm_score(int64_t n, const int32_t* tokens, const uint64_t* key, const uint64_t* ctx,
                  const uint32_t* pos, double* score, int32_t n_seg, const int64_t* seg_off, double* sums)
{
#pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < n; ++t)
        score[t] = orc_score_word(orc_word(key[t], ctx[t], pos[t], tokens[t], 1));
    if (!sums) return;
    if (!seg_off) { double S = 0.0; for (int64_t t = 0; t < n; ++t) S += score[t]; sums[0] = S; return; }
    for (int32_t g = 0; g < n_seg; ++g) {
        double S = 0.0;
        for (int64_t t = seg_off[g]; t < seg_off[g + 1]; ++t) S += score[t];
        sums[g] = S;
    }
}

/* ------------------------------------------------------------------ */
/* truncation before the race                                          */
/* ------------------------------------------------------------------ */

static int orc_double_desc(const void* a, const void* b)
{
    double x = *(const double*)a, y = *(const double*)b;
    return x > y ? -1 : (x < y ? 1 : 0);
}

static int orc_double_asc(const void* a, const void* b)
{
    return -orc_double_desc(a, b);
}

/* out[r*V + i] = l[i] if token i survives the truncation, -inf otherwise.
 *   top-k (top_k > 0): l_(k) is the k-th largest usable logit counting
 *     duplicates (usable: neither NaN nor -inf); a token is kept iff its logit
 *     is >= l_(k), so every token tied with l_(k) is kept.  With fewer than k
 *     usable tokens all usable tokens are kept.  top_k <= 0: all usable tokens.
 *   top-p (top_p < 1), on the top-k survivors with probabilities
 *     softmax(l / T) over them: walk the survivors in ascending logit order,
 *     adding each token's probability e_j / Z (e_j = exp((l_j - max l) / T),
 *     Z = the sum of the e_j taken in the same ascending order) to a running
 *     sum.  Tokens of equal logit form one group; a group is removed iff the
 *     running sum at its last token is <= 1 - top_p.  The group of the largest
 *     logit is always kept.  (For distinct logits this is the usual nucleus
 *     rule; a group is never split.)
 *   margin[r] (nullable): the smallest |running sum - (1 - top_p)| over the
 *     group ends (+inf without top-p), for flip accounting. */
void orc_truncate_rows(const float* logits, int64_t n_rows, int64_t V, int64_t stride, double T,
                       int32_t top_k, double top_p, float* out, double* margin)
{
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < n_rows; ++r) {
        const float* l = logits + r * stride;
        float* o = out + r * V;
        double* v = (double*)malloc(sizeof(double) * (size_t)(V > 0 ? V : 1));
        int64_t n = 0;
        for (int64_t i = 0; i < V; ++i)
            if (!isnan(l[i]) && l[i] != -INFINITY) v[n++] = (double)l[i];
        double cut = -INFINITY;
        if (top_k > 0 && n >= top_k) {
            qsort(v, (size_t)n, sizeof(double), orc_double_desc);
            cut = v[top_k - 1];
        }
        double mg = INFINITY;
        if (top_p < 1.0 && n > 0) {
            /* survivors of top-k, ascending */
            int64_t m = 0;
            for (int64_t i = 0; i < V; ++i)
                if (!isnan(l[i]) && l[i] != -INFINITY && (double)l[i] >= cut) v[m++] = (double)l[i];
            qsort(v, (size_t)m, sizeof(double), orc_double_asc);
            double top = v[m - 1], Z = 0.0;
            for (int64_t j = 0; j < m; ++j) Z += exp((v[j] - top) / T);
            double run = 0.0, keep_from = top;
            for (int64_t j = 0; j < m; ++j) {
                run += exp((v[j] - top) / T) / Z;
                int group_end = j + 1 == m || v[j + 1] != v[j];
                if (!group_end) continue;
                double d = fabs(run - (1.0 - top_p));
                if (d < mg) mg = d;
                if (v[j] == top) break;
                if (run <= 1.0 - top_p) keep_from = j + 1 < m ? v[j + 1] : top;
                else { keep_from = v[j]; break; }
            }
            /* the kept survivors are those with logit >= keep_from */
            if (keep_from > cut) cut = keep_from;
        }
        for (int64_t i = 0; i < V; ++i)
            o[i] = (!isnan(l[i]) && l[i] != -INFINITY && (double)l[i] >= cut) ? l[i] : -INFINITY;
        if (margin) margin[r] = mg;
        free(v);
    }
}

/* ------------------------------------------------------------------ */
/* detection scores and p-values                                       */
/* ------------------------------------------------------------------ */

/* kind 0 Aaronson, 1 U-score, 2 Li (param Delta), 3 Lattimore PL (param eps) */
double orc_score_kind(uint32_t w, int32_t kind, double param)
{
    double r = orc_uniform(w), one_minus_r = orc_one_minus_uniform(w);
    if (kind == 0) return orc_score_word(w);
    if (kind == 1) return r;
    if (kind == 2) {
        double k = floor(1.0 / (1.0 - param));
        double q = 1.0 - k * (1.0 - param);
        double ln_r = w < 0x80000000u ? log(r) : log1p(-one_minus_r);
        double sum = k * exp(ln_r * param / (1.0 - param));
        if (q > 0.0) sum += exp(ln_r * (1.0 - q) / q);
        return log(sum);
    }
    if (kind == 3) {
        double cap = 1.0 / sqrt(param), x = 1.0 / sqrt(one_minus_r);
        return (x < cap ? x : cap) - (2.0 - sqrt(param));
    }
    return NAN;
}

/* ln P(Gamma(M,1) >= S) = ln sum_{j=0}^{M-1} e^{-S} S^j / j!  (M >= 1), the terms
 * added in log space from j = 0 up.  The log-term ln(e^{-S} S^j / j!) is the
 * running sum -S + sum_{i<=j} (ln S - ln i), kept with Kahan's compensation: over
 * M ~ 10^7 additions to a value of size ~S its plain rounding would drift by
 * ~1e-6. */
double orc_gamma_tail_logp(int64_t M, double S)
{
    if (S <= 0.0) return 0.0;
    double lt = -S, comp = 0.0, ls = log(S), m = lt, acc = 1.0;  /* running log-sum-exp: m + ln acc */
    for (int64_t j = 1; j < M; ++j) {
        const double y = (ls - log((double)j)) - comp;
        const double t = lt + y;
        comp = (t - lt) - y;
        lt = t;
        if (lt > m) { acc = acc * exp(m - lt) + 1.0; m = lt; }
        else acc += exp(lt - m);
    }
    return m + log(acc);
}

static double orc_chernoff_exponent(double lambda, double M, double S)
{
    if (lambda == 0.0) return 0.0;
    return M * log(expm1(lambda) / lambda) - lambda * S;
}

/* min over lambda >= 0 of the Chernoff exponent (0 at lambda = 0); the
 * exponent is convex in lambda, so golden-section search on [0, L] with L
 * grown until the exponent rises */
double orc_chernoff_u_logp(int64_t M, double S)
{
    double Md = (double)M;
    if (S <= 0.5 * Md) return 0.0;
    if (S >= Md) return -INFINITY;
    double hi = 1.0;
    while (orc_chernoff_exponent(2.0 * hi, Md, S) < orc_chernoff_exponent(hi, Md, S) && hi < 1e6) hi *= 2.0;
    double lo = 0.0, up = 2.0 * hi;
    const double g = 0.6180339887498949;
    double a = up - g * (up - lo), b = lo + g * (up - lo);
    double fa = orc_chernoff_exponent(a, Md, S), fb = orc_chernoff_exponent(b, Md, S);
    for (int it = 0; it < 200; ++it) {
        if (fa < fb) { up = b; b = a; fb = fa; a = up - g * (up - lo); fa = orc_chernoff_exponent(a, Md, S); }
        else { lo = a; a = b; fa = fb; b = lo + g * (up - lo); fb = orc_chernoff_exponent(b, Md, S); }
    }
    double best = fa < fb ? fa : fb;
    return best < 0.0 ? best : 0.0;
}

/* Detector pass with a score kind: per token score (kind, param) of the
 * regenerated first-arrival word; per segment sums and log p-values
 * (kind 0: Gamma tail, kind 1: Chernoff bound on the U-score; NaN otherwise). */
void orc_wm_detect(int64_t n, const int32_t* tokens, const uint64_t* key, const uint64_t* ctx, const uint32_t* pos,
                   int32_t kind, double param, int32_t n_seg, const int64_t* seg_off, double* score, double* sums,
                   double* logp)
{
#pragma omp parallel for schedule(static)
    for (int64_t t = 0; t < n; ++t)
        score[t] = orc_score_kind(orc_word(key[t], ctx[t], pos[t], tokens[t], 1), kind, param);
#pragma omp parallel for schedule(dynamic, 16)
    for (int32_t g = 0; g < n_seg; ++g) {
        double S = 0.0;
        for (int64_t t = seg_off[g]; t < seg_off[g + 1]; ++t) S += score[t];
        sums[g] = S;
        int64_t M = seg_off[g + 1] - seg_off[g];
        if (!logp) continue;
        if (M == 0) logp[g] = 0.0;
        else if (kind == 0) logp[g] = orc_gamma_tail_logp(M, S);
        else if (kind == 1) logp[g] = orc_chernoff_u_logp(M, S);
        else logp[g] = NAN;
    }
}

/* ------------------------------------------------------------------ */
/* dynamic IID draft tree                                              */
/* ------------------------------------------------------------------ */

/* SplitMix64's output function (Steele, Lea, Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA'14) */
uint64_t orc_mix64(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

uint64_t orc_child_label(uint64_t parent, int32_t token)
{
    return orc_mix64(parent ^ ((uint64_t)(uint32_t)(token + 1) * 0x9E3779B97F4A7C15ull));
}

/* Fixed-capacity layout, per sequence b: node (d, i) = b*N1 + (d == 0 ? 0 :
 * 1 + (d-1)*K + i), N1 = 1 + K*gamma.  Draft rows depth-major: depth d's rows
 * start at D_d = n_seq*(d == 0 ? 0 : 1 + (d-1)*K); w_d = (d == 0 ? 1 : K) per
 * sequence; row (b, i) of the depth = b*w_d + i is draft row D_d + b*w_d + i,
 * owned by node (b, d, i).  A row with k = 0 is an
 * absent node.  For every present row (b, i) of depth d, its distinct draft
 * labels m < ndist (in list order) get child slots j = 0, 1, ... in row order
 * then list order; child j: ids (key, label(child), pos + 1), k = mult, its
 * node index written to child_node[draft row (d, i)][m] and its ids to the
 * node arrays; slots j >= the number of children get k = 0. */
void orc_tree_expand(int32_t n_seq, int32_t K, int32_t gamma, int32_t depth, const int32_t* tok,
                     const int32_t* mult, const int32_t* ndist, const uint64_t* key, const uint64_t* ctx,
                     const uint32_t* pos, const int32_t* row_k, uint64_t* next_key, uint64_t* next_ctx,
                     uint32_t* next_pos, int32_t* next_k, int32_t* child_node, uint64_t* node_key,
                     uint64_t* node_ctx, uint32_t* node_pos)
{
    int64_t N1 = 1 + (int64_t)K * gamma;
    int32_t w = depth == 0 ? 1 : K;
    int64_t D_d = depth == 0 ? 0 : (int64_t)n_seq * (1 + (int64_t)(depth - 1) * K);  /* first draft row of depth d */
    int64_t off_n = 1 + (int64_t)depth * K;                                          /* node offset of depth d+1 */
    for (int32_t b = 0; b < n_seq; ++b) {
        int32_t j = 0;
        for (int32_t i = 0; i < w; ++i) {
            int64_t r = (int64_t)b * w + i;
            int64_t dr = D_d + r;
            for (int32_t m = 0; m < K; ++m) child_node[dr * K + m] = -1;
            if (row_k[r] <= 0) continue;
            for (int32_t m = 0; m < ndist[r]; ++m) {
                int64_t q = (int64_t)b * K + j;
                next_key[q] = key[r];
                next_ctx[q] = orc_child_label(ctx[r], tok[r * K + m]);
                next_pos[q] = pos[r] + 1u;
                next_k[q] = mult[r * K + m];
                int64_t node = (int64_t)b * N1 + off_n + j;
                child_node[dr * K + m] = (int32_t)node;
                node_key[node] = next_key[q];
                node_ctx[node] = next_ctx[q];
                node_pos[node] = next_pos[q];
                ++j;
            }
        }
        for (; j < K; ++j) {
            int64_t q = (int64_t)b * K + j;
            next_key[q] = key[(int64_t)b * w];
            next_ctx[q] = 0;
            next_pos[q] = 0;
            next_k[q] = 0;
        }
    }
}

/* ------------------------------------------------------------------ */
/* non-identical proposals (App. A, heterogeneous proposals)           */
/* ------------------------------------------------------------------ */

/* The augmented race lives on V x [B] (blocks b = 0..B-1).  Its first
 * arrivals E_(i,b) are B independent Exp(1) per token, generated from three
 * keyed words by competing exponentials: the minimum of B iid Exp(1) is
 * Exp(B), it sits in a uniform block independent of its value, and the other
 * B-1 exceed it by independent Exp(1) amounts.  So, with E'_i the token's
 * usual first arrival,
 *     J_i     = floor(B * word(key ^ kBlockJ, i) / 2^32),
 *     E_(i,b) = E'_i / B                                      for b = J_i,
 *     E_(i,b) = E'_i / B + exp1(word(key ^ (b+1) kBlockF, i)) otherwise.
 * B = 1 gives E_(i,0) = E'_i, the identical-proposal source. */
#define ORC_BLOCK_J 0x3C6EF372FE94F82Bull
#define ORC_BLOCK_F 0xBB67AE8584CAA73Bull

int32_t orc_block_j(uint64_t key, uint64_t ctx, uint32_t pos, int64_t i, int32_t B)
{
    uint32_t w = orc_word(key ^ ORC_BLOCK_J, ctx, pos, i, 1);
    return (int32_t)(((uint64_t)w * (uint64_t)(uint32_t)B) >> 32);
}

double orc_block_e(uint64_t key, uint64_t ctx, uint32_t pos, int64_t i, int32_t b, int32_t B)
{
    double e = orc_exp1(orc_word(key, ctx, pos, i, 1)) / (double)B;
    if (b != orc_block_j(key, ctx, pos, i, B))
        e += orc_exp1(orc_word(key ^ ((uint64_t)(uint32_t)(b + 1) * ORC_BLOCK_F), ctx, pos, i, 1));
    return e;
}

/* Proposal b's sample at each row: X = argmin_i ln E_(i,b) - q_i/T over block
 * b (the race of Q~_b, which puts no mass outside block b); ties to the
 * smaller token.  x = -1 when no token is usable; margin = second-smallest
 * minus smallest key (+inf with fewer than two usable tokens). */
void orc_block_draft_rows(const float* q, int64_t n_rows, int64_t V, int64_t stride, double T, const uint64_t* key,
                          const uint64_t* ctx, const uint32_t* pos, const int32_t* block, int32_t B, int32_t* x,
                          double* key_out, double* margin)
{
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < n_rows; ++r) {
        double best = INFINITY, second = INFINITY;
        int64_t bi = -1;
        for (int64_t i = 0; i < V; ++i) {
            double l = (double)q[r * stride + i];
            if (isnan(l) || l == -INFINITY) continue;
            double k = log(orc_block_e(key[r], ctx[r], pos[r], i, block[r], B)) - l / T;
            if (bi < 0 || k < best) { second = best; best = k; bi = i; }
            else if (k < second) second = k;
        }
        x[r] = (int32_t)bi;
        if (key_out) key_out[r] = bi >= 0 ? best : INFINITY;
        if (margin) margin[r] = bi >= 0 && second < INFINITY ? second - best : INFINITY;
    }
}

/* One step with B proposals at each context c (rows p[c], q[c*B + b]):
 *   x[c*B + b]  = proposal b's sample (orc_block_draft_rows);
 *   (y[c], j[c]) = argmin over (i, b) of E_(i,b) / P~(i,b), P~(i,b) = p_i / B,
 *                  i.e. of ln E_(i,b) - p_i/T (the common ln B - ln Z drops out);
 *                  ties to the smaller i, then b;
 *   word[c]     = the watermark word of y: its usual first-arrival word, whose
 *                  E'_y = B E_(y,j) is the pivot a detector sees;
 *   accept[c]   = [y in {x[c*B + b]}];  margin_y = the target's key gap. */
void orc_hetero_rows(const float* p, const float* q, int64_t n_ctx, int32_t B, int64_t V, double T,
                     const uint64_t* key, const uint64_t* ctx, const uint32_t* pos, int32_t* x, int32_t* y,
                     int32_t* j, uint32_t* word, int32_t* accept, double* margin_y, double* margin_x)
{
    int64_t nr = n_ctx * B;
    uint64_t* rk = malloc((size_t)nr * sizeof(uint64_t));
    uint64_t* rc = malloc((size_t)nr * sizeof(uint64_t));
    uint32_t* rp = malloc((size_t)nr * sizeof(uint32_t));
    int32_t* rb = malloc((size_t)nr * sizeof(int32_t));
    for (int64_t r = 0; r < nr; ++r) {
        rk[r] = key[r / B];
        rc[r] = ctx[r / B];
        rp[r] = pos[r / B];
        rb[r] = (int32_t)(r % B);
    }
    orc_block_draft_rows(q, nr, V, V, T, rk, rc, rp, rb, B, x, NULL, margin_x);
    free(rk);
    free(rc);
    free(rp);
    free(rb);
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t c = 0; c < n_ctx; ++c) {
        double best = INFINITY, second = INFINITY;
        int64_t bi = -1;
        int32_t bb = -1;
        for (int64_t i = 0; i < V; ++i) {
            double l = (double)p[c * V + i];
            if (isnan(l) || l == -INFINITY) continue;
            for (int32_t b = 0; b < B; ++b) {
                double k = log(orc_block_e(key[c], ctx[c], pos[c], i, b, B)) - l / T;
                if (bi < 0 || k < best) { second = best; best = k; bi = i; bb = b; }
                else if (k < second) second = k;
            }
        }
        y[c] = (int32_t)bi;
        j[c] = bb;
        word[c] = bi >= 0 ? orc_word(key[c], ctx[c], pos[c], bi, 1) : 0u;
        int32_t acc = 0;
        for (int32_t b = 0; b < B; ++b) acc |= (bi >= 0 && x[c * B + b] == (int32_t)bi);
        accept[c] = acc;
        if (margin_y) margin_y[c] = bi >= 0 && second < INFINITY ? second - best : INFINITY;
    }
}

/* One depth of the draft tree of B proposals, each drafting a chain (the
 * proposition's one-step coupling applied at every node).  Layout of the
 * fixed-capacity tree, per sequence s: node (s, d, o) = s*N1 + (d == 0 ? 0 :
 * 1 + (d-1)*B + o), N1 = 1 + B*gamma; node lists depth-major, depth d's rows
 * from L_d = n_seq*(d == 0 ? 0 : 1 + (d-1)*B), w_d = (d == 0 ? 1 : B) per
 * sequence, node (s, d, o) owning list row L_d + s*w_d + o; proposal rows
 * (s, b) = s*B + b per depth.  A proposal at node o (owner[r]; -1 = stopped)
 * that drew token x (x < 0 stops it) moves to the child (d+1, f), f = the
 * smallest proposal at the same node that drew x.  Node o's list: the tokens
 * of the proposals b with first[b] = b at o, in increasing b, with child
 * (d+1, b).  Depth d+1's node (s, d+1, b) holds its identities iff b owns it
 * (zeros otherwise); next rows (key, label(c||x), pos + 1, f) for live
 * proposals, zeros and owner -1 for stopped ones (written when depth + 1 <
 * gamma). */
void orc_hetero_expand(int32_t n_seq, int32_t B, int32_t gamma, int32_t depth, const int32_t* tok,
                       const uint64_t* key, const uint64_t* ctx, const uint32_t* pos, const int32_t* owner,
                       uint64_t* next_key, uint64_t* next_ctx, uint32_t* next_pos, int32_t* next_owner,
                       int32_t* list_tok, int32_t* list_nd, int32_t* child_node, uint64_t* node_key,
                       uint64_t* node_ctx, uint32_t* node_pos)
{
    int64_t N1 = 1 + (int64_t)B * gamma;
    int32_t w = depth == 0 ? 1 : B;
    int64_t L_d = depth == 0 ? 0 : (int64_t)n_seq * (1 + (int64_t)(depth - 1) * B);
    int32_t alive[64], first[64];
    for (int64_t s = 0; s < n_seq; ++s) {
        const int64_t r0 = s * B;
        for (int32_t b = 0; b < B; ++b)
            alive[b] = owner[r0 + b] >= 0 && owner[r0 + b] < w && tok[r0 + b] >= 0;
        for (int32_t b = 0; b < B; ++b) {
            first[b] = -1;
            if (!alive[b]) continue;
            for (int32_t t = 0; t <= b; ++t)
                if (alive[t] && owner[r0 + t] == owner[r0 + b] && tok[r0 + t] == tok[r0 + b]) {
                    first[b] = t;
                    break;
                }
        }
        const int64_t child0 = s * N1 + 1 + (int64_t)depth * B;
        for (int32_t o = 0; o < w; ++o) {
            const int64_t lr = L_d + s * w + o;
            int32_t m = 0;
            for (int32_t t = 0; t < B; ++t)
                if (alive[t] && owner[r0 + t] == o && first[t] == t) {
                    list_tok[lr * B + m] = tok[r0 + t];
                    child_node[lr * B + m] = (int32_t)(child0 + t);
                    ++m;
                }
            list_nd[lr] = m;
            for (; m < B; ++m) {
                list_tok[lr * B + m] = -1;
                child_node[lr * B + m] = -1;
            }
        }
        for (int32_t b = 0; b < B; ++b) {
            const int64_t r = r0 + b;
            uint64_t k = 0, lab = 0;
            uint32_t p = 0;
            if (alive[b]) {
                k = key[r];
                lab = orc_child_label(ctx[r], tok[r]);
                p = pos[r] + 1u;
            }
            const int owns = alive[b] && first[b] == b;
            node_key[child0 + b] = owns ? k : 0;
            node_ctx[child0 + b] = owns ? lab : 0;
            node_pos[child0 + b] = owns ? p : 0u;
            if (depth + 1 < gamma) {
                next_key[r] = k;
                next_ctx[r] = lab;
                next_pos[r] = p;
                next_owner[r] = alive[b] ? first[b] : -1;
            }
        }
    }
}

/*
 * The LM head (the last layer that produces the logits the race reads): the
 * inner product of each context's hidden state with each token's row of the
 * LM-head matrix, logits[r][i] = sum_j hidden[r][j] * weight[i][j], summed in
 * fp64 in index order.  The operands are the fp32 images of bf16 values, so
 * every product is exact in fp64; for operands whose partial sums are exactly
 * representable (small dyadic values) the result is exact in any order.
 */
void orc_lmhead_logits(const float* hidden, const float* weight, int64_t n_rows, int64_t V, int64_t d,
                       double* out)
{
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < n_rows; ++r)
        for (int64_t i = 0; i < V; ++i) {
            double acc = 0.0;
            for (int64_t j = 0; j < d; ++j) acc += (double)hidden[r * d + j] * (double)weight[i * d + j];
            out[r * V + i] = acc;
        }
}

/* raw words of rows x vocab for a given arrival (bit-exact checks) */
void orc_words(int64_t n_rows, int64_t V, const uint64_t* key, const uint64_t* ctx, const uint32_t* pos,
               int32_t arrival, uint32_t* out)
{
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < n_rows; ++r)
        for (int64_t i = 0; i < V; ++i) out[r * V + i] = orc_word(key[r], ctx[r], pos[r], i, arrival);
}

int orc_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
    return omp_get_max_threads();
#else
    (void)n;
    return 1;
#endif
}
