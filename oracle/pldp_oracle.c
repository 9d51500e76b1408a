/*
 * pldp_oracle.c -- plain, slow, single-threaded CPU oracle of the PLD+
 * drafting and greedy verification step (PLD+, arXiv 2412.01447).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the independent reference that the
 * CUDA library is checked against.  It shares no code, header, helper or
 * constant generator with the CUDA path, and the CUDA path never calls it.
 * Only the test-suite, the smoke check and the CPU-baseline leg of the
 * benchmark may load it.
 *
 * Every floating-point quantity is carried in double precision.  bf16 and
 * fp32 inputs convert to double exactly, so every product of two inputs is
 * exact and the only rounding is in the sums (over at most a few thousand
 * terms) and in the final division/sqrt of the cosine.
 *
 * Indexing: all positions are 0-based.  For sequence b with length
 * L = seq_len[b], the last token is x_t with t = L - 1.  The artifacts (hidden
 * rows and attention rows) exist for positions 0..t-1 only, because the
 * forward pass that will produce position t's artifacts has not run yet
 * (Sec. 4.2.2 notes that x_t has no hidden state at drafting time).
 *
 * Readings of passages the paper leaves silent, garbled or ambiguous are
 * marked READING below; each one is listed in the design notes.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* Status bits written into status[b] (OR-ed in; the caller clears them).
 * These numeric values are part of the library's documented interface and
 * are restated here, not shared. */
#define ORC_ST_CAND_OVERFLOW 1u  /* more candidates than C_cap            */
#define ORC_ST_TOKEN_RANGE   2u  /* a draft token outside [0, V)          */
#define ORC_ST_CAPACITY      4u  /* append would exceed T_cap: no append  */
#define ORC_ST_SEQ_LEN       8u  /* seq_len outside [0, T_cap] (or < 1)   */
#define ORC_ST_DRAFT_LEN    16u  /* draft_len outside [0, K]: clamped     */
#define ORC_ST_ROW_INDEX    32u  /* selected row outside [0, R): ignored  */

#define ORC_F32  0
#define ORC_BF16 1
#define ORC_AGG_MAX 0
#define ORC_AGG_SUM 1

/* Exact widening of one stored element to double. */
static double orc_load(const void* base, int dtype, int64_t idx) {
    if (dtype == ORC_F32) {
        return (double)((const float*)base)[idx];
    } else {
        uint16_t h = ((const uint16_t*)base)[idx];
        uint32_t bits = ((uint32_t)h) << 16;   /* bf16 is the top half of fp32 */
        float f;
        memcpy(&f, &bits, sizeof f);
        return (double)f;
    }
}

/* --------------------------------------------------------------------------
 * Candidate search.  Eq. 1 (Sec. 4.2, Drafting Algorithm):
 *     P = { j | x_j = x_t, j < t }.
 * READING (n-gram): following the prompt-lookup heritage that PLD+ builds on
 * (Sec. 2 and Fig. 2: PLD drafts from the earlier occurrence that agrees with
 * the context on the most tokens), the match is on the longest suffix n-gram
 * that occurs earlier:
 * for n = n_max down to n_min, P_n = { j < t : j-n+1 >= 0 and
 * x_{j-k} = x_{t-k} for k = 0..n-1 }; the first non-empty P_n is P and its n
 * is match_len.  n_min = n_max = 1 is Eq. 1 itself.
 * P is listed in ascending order; the true |P| is reported even when only the
 * first C_cap positions fit.
 * ------------------------------------------------------------------------ */
static int orc_ngram_matches(const int32_t* x, int64_t j, int64_t t, int n) {
    if (j - (n - 1) < 0) return 0;
    for (int k = 0; k < n; ++k)
        if (x[j - k] != x[t - k]) return 0;
    return 1;
}

int pldpo_find_candidates(const int32_t* ids, int64_t ids_stride,
                          const int32_t* seq_len, int B, int64_t T_cap,
                          int ngram_min, int ngram_max,
                          int32_t* cand_pos, int C_cap,
                          int32_t* cand_count, int32_t* match_len,
                          uint32_t* status) {
    if (B < 0 || ngram_min < 1 || ngram_max < ngram_min || C_cap < 0) return 1;
    for (int b = 0; b < B; ++b) {
        const int32_t* x = ids + (int64_t)b * ids_stride;
        int64_t L = seq_len[b];
        cand_count[b] = 0;
        match_len[b] = 0;
        if (L < 0 || L > T_cap) {
            if (status) status[b] |= ORC_ST_SEQ_LEN;
            continue;
        }
        int64_t t = L - 1;
        if (t < 1) continue;                    /* no j < t exists */
        for (int n = ngram_max; n >= ngram_min; --n) {
            int64_t count = 0;
            for (int64_t j = 0; j < t; ++j) {
                if (orc_ngram_matches(x, j, t, n)) {
                    if (count < C_cap) cand_pos[(int64_t)b * C_cap + count] = (int32_t)j;
                    ++count;
                }
            }
            if (count > 0) {
                cand_count[b] = (int32_t)count;
                match_len[b] = n;
                if (count > C_cap && status) status[b] |= ORC_ST_CAND_OVERFLOW;
                break;
            }
        }
    }
    return 0;
}

/* --------------------------------------------------------------------------
 * Ranking by hidden states.  Eq. 3 (Sec. 4.2.2):
 *     j* = argmax_{j in P} cos_sim(H_{j-1}, H_{t-1})
 * on the caller-chosen layer l, whose [T_cap, d] slice per sequence is passed.
 * Optional threshold (App. B.3): j is kept only if cos > theta (strict).
 * READING: j = 0 has no H_{-1}; it is not eligible and scores -inf.
 * READING: a zero-norm vector gives cos = 0 (no epsilon otherwise).
 * READING: ties go to the smallest position j.
 * scores[b*C_cap + i] is the score of the i-th listed candidate.
 * A seq_len outside [0, T_cap] skips the sequence (SEQ_LEN, best_pos = -1).
 * ------------------------------------------------------------------------ */
static double orc_cosine(const void* H, int dtype, int64_t row_a, int64_t row_b, int64_t d) {
    double dot = 0.0, na = 0.0, nb = 0.0;
    for (int64_t k = 0; k < d; ++k) {
        double a = orc_load(H, dtype, row_a + k);
        double c = orc_load(H, dtype, row_b + k);
        dot += a * c;
        na += a * a;
        nb += c * c;
    }
    if (na == 0.0 || nb == 0.0) return 0.0;
    return dot / sqrt(na * nb);
}

int pldpo_rank_hidden(const void* H, int dtype, int64_t d, int64_t seq_stride,
                      const int32_t* seq_len, int B, int64_t T_cap,
                      const int32_t* cand_pos, const int32_t* cand_count, int C_cap,
                      double threshold, double* scores,
                      int32_t* best_pos, double* best_score, uint32_t* status) {
    if (B < 0 || d < 1 || C_cap < 0 || (dtype != ORC_F32 && dtype != ORC_BF16)) return 1;
    for (int b = 0; b < B; ++b) {
        if (seq_len[b] < 0 || seq_len[b] > T_cap) {         /* sequence skipped */
            if (status) status[b] |= ORC_ST_SEQ_LEN;
            best_pos[b] = -1;
            if (best_score) best_score[b] = -INFINITY;
            continue;
        }
        int64_t t = (int64_t)seq_len[b] - 1;
        int64_t n = cand_count[b] < 0 ? 0 : cand_count[b];
        if (n > C_cap) n = C_cap;
        int32_t bj = -1;
        double bs = -INFINITY;
        for (int64_t i = 0; i < n; ++i) {
            int64_t j = cand_pos[(int64_t)b * C_cap + i];
            double s = -INFINITY;
            if (j >= 1 && j < t) {
                int64_t row_cand  = (int64_t)b * seq_stride + (j - 1) * d;   /* H_{j-1} */
                int64_t row_query = (int64_t)b * seq_stride + (t - 1) * d;   /* H_{t-1} */
                s = orc_cosine(H, dtype, row_cand, row_query, d);
            }
            if (scores) scores[(int64_t)b * C_cap + i] = s;
            if (j >= 1 && j < t && s > threshold) {
                if (bj < 0 || s > bs || (s == bs && j < bj)) { bs = s; bj = (int32_t)j; }
            }
        }
        best_pos[b] = bj;
        if (best_score) best_score[b] = bj >= 0 ? bs : -INFINITY;
    }
    return 0;
}

/* --------------------------------------------------------------------------
 * Ranking by averaged hidden states -- the variant of Eq. 3 studied in App. B.2:
 * every hidden state is replaced by the mean of the m rows ending at it,
 *     Hbar_p = mean(H_{max(0, p-m+1)}, ..., H_p),
 * and candidate j scores cos(Hbar_{j-1}, Hbar_{t-1}).  m = 1 is Eq. 3.
 * READING: the printed formula averages H_1..H_m, the same rows for every
 * position; it is read as the window of the m positions ending at the position
 * averaged, cut at position 0 (fewer rows near the start).
 * Eligibility, zero norms, ties, the threshold and scores as pldpo_rank_hidden.
 * ------------------------------------------------------------------------ */
static void orc_window_mean(const void* H, int dtype, int64_t base, int64_t p, int m, int64_t d,
                            double* out) {
    int64_t lo = p - m + 1;
    if (lo < 0) lo = 0;
    for (int64_t k = 0; k < d; ++k) out[k] = 0.0;
    for (int64_t r = lo; r <= p; ++r)
        for (int64_t k = 0; k < d; ++k) out[k] += orc_load(H, dtype, base + r * d + k);
    for (int64_t k = 0; k < d; ++k) out[k] /= (double)(p - lo + 1);
}

int pldpo_rank_hidden_avg(const void* H, int dtype, int64_t d, int64_t seq_stride, int m,
                          const int32_t* seq_len, int B, int64_t T_cap,
                          const int32_t* cand_pos, const int32_t* cand_count, int C_cap,
                          double threshold, double* scores,
                          int32_t* best_pos, double* best_score, uint32_t* status) {
    if (B < 0 || d < 1 || m < 1 || C_cap < 0 || (dtype != ORC_F32 && dtype != ORC_BF16)) return 1;
    double* qv = (double*)malloc(sizeof(double) * (size_t)d);
    double* cv = (double*)malloc(sizeof(double) * (size_t)d);
    if (!qv || !cv) { free(qv); free(cv); return 2; }
    for (int b = 0; b < B; ++b) {
        if (seq_len[b] < 0 || seq_len[b] > T_cap) {         /* sequence skipped */
            if (status) status[b] |= ORC_ST_SEQ_LEN;
            best_pos[b] = -1;
            if (best_score) best_score[b] = -INFINITY;
            continue;
        }
        int64_t t = (int64_t)seq_len[b] - 1;
        int64_t n = cand_count[b] < 0 ? 0 : cand_count[b];
        if (n > C_cap) n = C_cap;
        int64_t base = (int64_t)b * seq_stride;
        if (t >= 1) orc_window_mean(H, dtype, base, t - 1, m, d, qv);     /* Hbar_{t-1} */
        int32_t bj = -1;
        double bs = -INFINITY;
        for (int64_t i = 0; i < n; ++i) {
            int64_t j = cand_pos[(int64_t)b * C_cap + i];
            double s = -INFINITY;
            if (j >= 1 && j < t) {
                orc_window_mean(H, dtype, base, j - 1, m, d, cv);         /* Hbar_{j-1} */
                double dot = 0.0, na = 0.0, nq = 0.0;
                for (int64_t k = 0; k < d; ++k) {
                    dot += cv[k] * qv[k];
                    na += cv[k] * cv[k];
                    nq += qv[k] * qv[k];
                }
                s = (na == 0.0 || nq == 0.0) ? 0.0 : dot / sqrt(na * nq);
            }
            if (scores) scores[(int64_t)b * C_cap + i] = s;
            if (j >= 1 && j < t && threshold < s) {           /* eligible: the smallest j wins a tie */
                if (bj < 0 || s > bs || (s == bs && j < bj)) { bs = s; bj = (int32_t)j; }
            }
        }
        best_pos[b] = bj;
        if (best_score) best_score[b] = bj >= 0 ? bs : -INFINITY;
    }
    free(qv);
    free(cv);
    return 0;
}

/* --------------------------------------------------------------------------
 * Ranking by attentions.  Eq. 2 (Sec. 4.2.1):
 *     j* = argmax_{j in P} max_{l in L*, g in G*} A^{(l,g)}_{t-1}
 * A holds, per sequence, the attention-probability rows of query t-1 for the
 * caller's R (layer, head) pairs: element (r, j) at
 *     A[b*seq_stride + r*row_stride + j].
 * row_idx (nullable) selects n_sel of the R rows (G* x L*); NULL = all R.
 * READING: the key index missing from Eq. 2 is the candidate j itself (the
 * induction-head target: query t-1 attends to the token that follows an
 * earlier occurrence of x_{t-1}, i.e. to the copied token x_j).
 * agg = SUM aggregates by summation instead (the Sec. 7.1 variant).
 * Ties go to the smallest j.  Candidates outside [0, t) score -inf and are
 * not eligible.  Selected rows outside [0, R) are left out (ROW_INDEX).
 * A seq_len outside [0, T_cap] skips the sequence (SEQ_LEN, best_pos = -1).
 * ------------------------------------------------------------------------ */
int pldpo_rank_attention(const void* A, int dtype, int R, int64_t row_stride, int64_t seq_stride,
                         const int32_t* row_idx, int n_sel, int agg,
                         const int32_t* seq_len, int B, int64_t T_cap,
                         const int32_t* cand_pos, const int32_t* cand_count, int C_cap,
                         double* scores, int32_t* best_pos, double* best_score, uint32_t* status) {
    if (B < 0 || R < 1 || C_cap < 0 || (dtype != ORC_F32 && dtype != ORC_BF16)) return 1;
    if (agg != ORC_AGG_MAX && agg != ORC_AGG_SUM) return 1;
    int rows = row_idx ? n_sel : R;
    if (rows < 1) return 1;
    int bad_rows = 0;
    for (int k = 0; k < rows; ++k) {
        int r = row_idx ? row_idx[k] : k;
        if (r < 0 || r >= R) bad_rows = 1;      /* such rows are left out of the aggregate */
    }
    for (int b = 0; b < B; ++b) {
        if (seq_len[b] < 0 || seq_len[b] > T_cap) {         /* sequence skipped */
            if (status) status[b] |= ORC_ST_SEQ_LEN;
            best_pos[b] = -1;
            if (best_score) best_score[b] = -INFINITY;
            continue;
        }
        if (bad_rows && status) status[b] |= ORC_ST_ROW_INDEX;
        int64_t t = (int64_t)seq_len[b] - 1;
        int64_t n = cand_count[b] < 0 ? 0 : cand_count[b];
        if (n > C_cap) n = C_cap;
        int32_t bj = -1;
        double bs = -INFINITY;
        for (int64_t i = 0; i < n; ++i) {
            int64_t j = cand_pos[(int64_t)b * C_cap + i];
            double s = -INFINITY;
            if (j >= 0 && j < t) {
                s = (agg == ORC_AGG_MAX) ? -INFINITY : 0.0;
                for (int k = 0; k < rows; ++k) {
                    int r = row_idx ? row_idx[k] : k;
                    if (r < 0 || r >= R) continue;
                    double a = orc_load(A, dtype, (int64_t)b * seq_stride + (int64_t)r * row_stride + j);
                    if (agg == ORC_AGG_MAX) { if (a > s) s = a; }
                    else s += a;
                }
            }
            if (scores) scores[(int64_t)b * C_cap + i] = s;
            if (j >= 0 && j < t) {
                if (bj < 0 || s > bs || (s == bs && j < bj)) { bs = s; bj = (int32_t)j; }
            }
        }
        best_pos[b] = bj;
        if (best_score) best_score[b] = bj >= 0 ? bs : -INFINITY;
    }
    return 0;
}

/* --------------------------------------------------------------------------
 * Draft prediction (Sec. 4.3):  xhat_i = x_{j*+i}, i = 1..K.
 * READING: the span stops at the last token x_t, so the draft has
 * d = min(K, t - j*) tokens; the rest of draft[b, :] is -1.  No candidate
 * (j* < 0), j* outside [0, t) or a seq_len beyond T_cap gives d = 0.
 * ------------------------------------------------------------------------ */
int pldpo_extract_draft(const int32_t* ids, int64_t ids_stride, const int32_t* seq_len,
                        int64_t T_cap, const int32_t* best_pos, int B, int K,
                        int32_t* draft, int32_t* draft_len) {
    if (B < 0 || K < 1) return 1;
    for (int b = 0; b < B; ++b) {
        int64_t t = (int64_t)seq_len[b] - 1;
        int64_t js = best_pos[b];
        int64_t d = 0;
        if (seq_len[b] <= T_cap && js >= 0 && js < t) d = (t - js < K) ? (t - js) : K;
        for (int64_t i = 0; i < K; ++i)
            draft[(int64_t)b * K + i] = (i < d) ? ids[(int64_t)b * ids_stride + js + 1 + i] : -1;
        draft_len[b] = (int32_t)d;
    }
    return 0;
}

/* --------------------------------------------------------------------------
 * Induction-head identification (Sec. 4.2.1): for generated tokens that also
 * occur earlier, find the position r* they were most likely copied from, and
 * count, for every (layer, head) row, how often that row puts its maximum
 * attention on r*.  The rows with the highest counts are the G* / L* of Eq. 2.
 *
 * Observation b: the generated token is x_p with p = pos[b]; ids[b, 0..p] is
 * the context; A holds, per observation, the R attention rows of query p-1 over
 * keys 0..p-1: element (r, key) at A[b*seq_stride + r*row_stride + key].
 *   P      = {j < p : x_j = x_p}
 *   ov(j)  = the largest k <= max_suffix with x_{j-i} = x_{p-i} for i < k
 *            (the overlapping suffix of the context before j and the output)
 *   r*     = argmax_{j in P} ov(j)
 *   row r counts when argmax_{key < p} A[r, key] = r*.
 * READING: ties in ov(j) go to the smallest j (the library's tie rule); ties in
 * a row's maximum go to the smallest key; Sec. 4.2.1's condition that the
 * attention peaks at position r* is applied to each row on its own (a row
 * counts when r* is the argmax of that head's row).
 * r_star[b] = r*, or -1 when P is empty (then nothing is counted); counts[r]
 * are ADDED to (uint32, caller-initialised) so that batches accumulate.
 * pos[b] outside [1, T_cap - 1] sets SEQ_LEN and counts nothing.
 * ------------------------------------------------------------------------ */
int pldpo_identify_heads(const int32_t* ids, int64_t ids_stride, const int32_t* pos, int B,
                         int64_t T_cap, int max_suffix, const void* A, int dtype, int R,
                         int64_t row_stride, int64_t seq_stride, uint32_t* counts,
                         int32_t* r_star, uint32_t* status) {
    if (B < 0 || R < 1 || max_suffix < 1 || (dtype != ORC_F32 && dtype != ORC_BF16)) return 1;
    for (int b = 0; b < B; ++b) {
        int64_t p = pos[b];
        if (r_star) r_star[b] = -1;
        if (p < 1 || p >= T_cap) {
            if (status) status[b] |= ORC_ST_SEQ_LEN;
            continue;
        }
        const int32_t* x = ids + (int64_t)b * ids_stride;
        int64_t rs = -1, best_ov = 0;
        for (int64_t j = 0; j < p; ++j) {
            if (x[j] != x[p]) continue;
            int64_t k = 0;
            while (k < max_suffix && j - k >= 0 && x[j - k] == x[p - k]) ++k;
            if (k > best_ov) { best_ov = k; rs = j; }     /* strict: the smallest j keeps a tie */
        }
        if (r_star) r_star[b] = (int32_t)rs;
        if (rs < 0) continue;
        for (int r = 0; r < R; ++r) {
            int64_t row = (int64_t)b * seq_stride + (int64_t)r * row_stride;
            double mx = orc_load(A, dtype, row);
            int64_t arg = 0;
            for (int64_t key = 1; key < p; ++key) {
                double v = orc_load(A, dtype, row + key);
                if (v > mx) { mx = v; arg = key; }
            }
            if (arg == rs) counts[r] += 1u;
        }
    }
    return 0;
}

/* Acceptance and bookkeeping shared by both verifications, for sequence b
 * whose K+1 target tokens (argmax or sampled) are tok[0..K]:
 * n = first i < d with draft_i != tok_i (else d), bonus = tok_n, then the
 * optional append to ids / seq_len and kv_keep_len = L + n.  Sec. 4.4. */
static void orc_accept(int b, int K, int V, const int32_t* tok, const int32_t* draft,
                       const int32_t* draft_len, int32_t* accept_len, int32_t* next_token,
                       int32_t* ids, int64_t ids_stride, int32_t* seq_len, int64_t T_cap,
                       int32_t* kv_keep_len, uint32_t* status) {
    int64_t d = draft_len[b];
    if (d < 0 || d > K) {
        if (status) status[b] |= ORC_ST_DRAFT_LEN;
        d = d < 0 ? 0 : K;
    }
    for (int64_t i = 0; i < d; ++i) {
        int32_t t = draft[(int64_t)b * K + i];
        if ((t < 0 || t >= V) && status) status[b] |= ORC_ST_TOKEN_RANGE;
    }
    int64_t n = d;
    for (int64_t i = 0; i < d; ++i) {
        if (draft[(int64_t)b * K + i] != tok[i]) { n = i; break; }
    }
    int32_t bonus = tok[n];
    accept_len[b] = (int32_t)n;
    next_token[b] = bonus;
    if (!seq_len) return;
    int64_t L = seq_len[b];
    if (L < 1 || L > T_cap) {
        if (status) status[b] |= ORC_ST_SEQ_LEN;
        if (kv_keep_len) kv_keep_len[b] = -1;
        return;
    }
    if (kv_keep_len) kv_keep_len[b] = (int32_t)(L + n);
    if (L + n + 1 > T_cap) {
        if (status) status[b] |= ORC_ST_CAPACITY;
        return;
    }
    if (ids) {
        int32_t* x = ids + (int64_t)b * ids_stride;
        for (int64_t i = 0; i < n; ++i) x[L + i] = draft[(int64_t)b * K + i];
        x[L + n] = bonus;
    }
    seq_len[b] = (int32_t)(L + n + 1);
}

/* --------------------------------------------------------------------------
 * Greedy verification (Sec. 4.4 with T = 0, and Sec. 3: one forward pass on
 * the draft gives K+1 distributions).  Row i of logits[b] is the target
 * model's distribution for the token after the first i draft tokens.
 *   a_i = argmax_v logits[b, i, v]   (first index among equal maxima)
 *   n   = first i < d with draft_i != a_i, else d       (accepted length)
 *   bonus = a_n                                          (next token)
 * Everything after the first mismatch is discarded.
 * Optional bookkeeping, when seq_len is given: kv_keep_len[b] = L + n with
 * L the old seq_len (x_t and the n accepted tokens are the positions whose
 * keys/values the verifying forward pass computed and that survive); then
 * draft_0..draft_{n-1}, bonus are appended to ids (when given) at L..L+n and
 * seq_len[b] = L + n + 1.  An append that would pass T_cap changes neither
 * ids nor seq_len and sets CAPACITY.
 * ------------------------------------------------------------------------ */
int pldpo_verify_greedy(const void* logits, int dtype, int B, int K, int V,
                        const int32_t* draft, const int32_t* draft_len,
                        int32_t* argmax, int32_t* accept_len, int32_t* next_token,
                        int32_t* ids, int64_t ids_stride, int32_t* seq_len, int64_t T_cap,
                        int32_t* kv_keep_len, uint32_t* status) {
    if (B < 0 || K < 1 || V < 1 || (dtype != ORC_F32 && dtype != ORC_BF16)) return 1;
    if ((ids || kv_keep_len) && !seq_len) return 1;
    int32_t* av = (int32_t*)malloc(sizeof(int32_t) * (size_t)(K + 1));
    if (!av) return 2;
    for (int b = 0; b < B; ++b) {
        for (int i = 0; i <= K; ++i) {
            int64_t row = ((int64_t)b * (K + 1) + i) * (int64_t)V;
            double best = orc_load(logits, dtype, row);
            int32_t bi = 0;
            for (int64_t v = 1; v < V; ++v) {
                double x = orc_load(logits, dtype, row + v);
                if (x > best) { best = x; bi = (int32_t)v; }   /* strict: first max kept */
            }
            av[i] = bi;
            if (argmax) argmax[(int64_t)b * (K + 1) + i] = bi;
        }
        orc_accept(b, K, V, av, draft, draft_len, accept_len, next_token, ids, ids_stride,
                   seq_len, T_cap, kv_keep_len, status);
    }
    free(av);
    return 0;
}

/*
 * Sampling verification -- Sec. 4.4 at temperature T > 0 (the paper's sampled
 * runs use T = 1, Table 2): at each of the K+1 positions a token is drawn from
 * p = softmax(logits / T), and the draft is accepted up to the first position
 * whose drawn token differs from it; the token drawn there is the bonus.  For a
 * draft that is a single token per position (as PLD+'s is), this accepts token
 * i with probability p(draft_i) and, on a rejection, draws the bonus from p
 * restricted to the other tokens: exactly what sampling from the target alone
 * would emit.
 *
 * The random numbers are the caller's: position i of sequence b takes
 * u = uniforms[b, i] and draws the smallest v whose cumulative probability
 * sum_{v' <= v} p_v' exceeds u (inverse-CDF sampling).
 * READING: u outside [0, 1) is clamped into it; the paper does not say how its
 * samples are drawn, only that they are.
 * Finite logits only.  Probabilities are carried in double precision: with
 * m the row maximum, w_v = exp((l_v - m) / T), Z = sum w_v, and the draw is the
 * first v with sum_{v' <= v} w_v' > u * Z.
 */
int pldpo_verify_sample(const void* logits, int dtype, int B, int K, int V, double temperature,
                        const float* uniforms, const int32_t* draft, const int32_t* draft_len,
                        int32_t* sampled, int32_t* accept_len, int32_t* next_token,
                        int32_t* ids, int64_t ids_stride, int32_t* seq_len, int64_t T_cap,
                        int32_t* kv_keep_len, uint32_t* status) {
    if (B < 0 || K < 1 || V < 1 || (dtype != ORC_F32 && dtype != ORC_BF16)) return 1;
    if (!(temperature > 0.0) || isinf(temperature)) return 1;
    if ((ids || kv_keep_len) && !seq_len) return 1;
    int32_t* yv = (int32_t*)malloc(sizeof(int32_t) * (size_t)(K + 1));
    if (!yv) return 2;
    for (int b = 0; b < B; ++b) {
        for (int i = 0; i <= K; ++i) {
            int64_t row = ((int64_t)b * (K + 1) + i) * (int64_t)V;
            double m = orc_load(logits, dtype, row);
            for (int64_t v = 1; v < V; ++v) {
                double x = orc_load(logits, dtype, row + v);
                if (x > m) m = x;
            }
            double Z = 0.0;
            for (int64_t v = 0; v < V; ++v) Z += exp((orc_load(logits, dtype, row + v) - m) / temperature);
            double u = (double)uniforms[(int64_t)b * (K + 1) + i];
            if (!(u >= 0.0)) u = 0.0;                                 /* also NaN */
            if (u >= 1.0) u = nextafter(1.0, 0.0);
            double target = u * Z, c = 0.0;
            int32_t y = -1, last_pos = 0;
            for (int64_t v = 0; v < V; ++v) {
                double w = exp((orc_load(logits, dtype, row + v) - m) / temperature);
                if (w > 0.0) last_pos = (int32_t)v;
                c += w;
                if (c > target) { y = (int32_t)v; break; }
            }
            if (y < 0) y = last_pos;     /* unreachable: the sum ends at Z > u * Z */
            yv[i] = y;
            if (sampled) sampled[(int64_t)b * (K + 1) + i] = y;
        }
        orc_accept(b, K, V, yv, draft, draft_len, accept_len, next_token, ids, ids_stride,
                   seq_len, T_cap, kv_keep_len, status);
    }
    free(yv);
    return 0;
}

int pldpo_version(void) { return 1; }
