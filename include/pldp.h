/*
 * pldp.h -- C ABI of the GB300 (sm_103a) PLD+ drafting and greedy
 * verification library.
 *
 * PLD+ (arXiv 2412.01447) speeds up decoding of input-guided tasks by
 * drafting a span copied from the context and verifying it with one forward
 * pass of the target model.  Per decode step and per sequence this library:
 *
 *   1. finds the earlier occurrences P of the last token (Eq. 1), narrowed to
 *      the longest suffix n-gram that occurs earlier     -> pldp_find_candidates
 *   2. ranks P with a model artifact: the cosine between hidden states
 *      H_{j-1} and H_{t-1} (Eq. 3)                        -> pldp_rank_hidden
 *      or the max attention of query t-1 over selected
 *      (layer, head) rows (Eq. 2)                         -> pldp_rank_attention
 *   3. drafts the K tokens after the best occurrence j*
 *      (Sec. 4.3)                                         -> pldp_extract_draft
 *   4. verifies the draft greedily against the target
 *      model's K+1 next-token distributions (Sec. 4.4)    -> pldp_verify_greedy
 *      or by sampling at temperature T                    -> pldp_verify_sample
 *
 * Fused forms: pldp_draft_step runs 1-3 in one launch (scanning the contexts, or
 * with the incremental token index of pldp_index_build); pldp_verify_greedy_draft
 * and pldp_verify_sample_draft run 4 (greedy or by sampling) for the current step
 * and then 1-3 for the next step.  Offline:
 * pldp_rank_hidden_avg (App. B.2) and pldp_identify_heads / pldp_top_heads
 * (Sec. 4.2.1).
 *
 * Conventions shared by every call
 *  - Every pointer argument is a DEVICE pointer owned by the caller (the
 *    attention rows A of the ranking calls may also be device-addressable
 *    page-locked host memory, read in place); the
 *    library allocates nothing and keeps no state between calls, except the
 *    caller-provided verification workspace described at pldp_verify_greedy,
 *    the caller-provided token index that the indexed drafting calls keep up
 *    to date, and the fixed scratch area of pldp_verify_greedy_noalloc.
 *  - All work is enqueued asynchronously on `stream` (a cudaStream_t; NULL is
 *    the legacy default stream).  No call synchronises the device or reads
 *    device memory on the host, so every call may be captured in a CUDA graph.
 *  - Positions are 0-based int32.  Sequence b holds seq_len[b] tokens in
 *    ids[b*ids_stride + 0 .. seq_len[b]-1]; its last token is x_t with
 *    t = seq_len[b] - 1.  Model artifacts exist for positions 0..t-1 only.
 *  - Host-side argument checks run before anything is enqueued; a failed
 *    check returns PLDP_ERR_INVALID_ARG (or PLDP_ERR_UNSUPPORTED) and
 *    enqueues nothing.  A CUDA launch failure returns PLDP_ERR_CUDA.
 *    pldp_last_error() then gives a message (per host thread).
 *  - Data-dependent problems found on the device never trap: they set bits in
 *    the optional per-sequence status word (uint32 status[B], OR-ed in; the
 *    caller clears it) and the call produces the documented fallback.
 *  - dtype PLDP_BF16 data is raw bfloat16; PLDP_F32 is IEEE float.  Inputs
 *    must be finite (NaN is not supported).
 *  - Calls that overlap on the device must not share output buffers.
 */
#ifndef PLDP_H
#define PLDP_H

#include <stddef.h>
#include <stdint.h>

#if defined(_WIN32)
#define PLDP_API
#else
#define PLDP_API __attribute__((visibility("default")))
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    PLDP_OK = 0,
    PLDP_ERR_INVALID_ARG = 1, /* null/misaligned pointer, bad size or stride  */
    PLDP_ERR_UNSUPPORTED = 2, /* dtype or size the kernels do not handle      */
    PLDP_ERR_CUDA = 3,        /* launch failed; see pldp_last_error()         */
    PLDP_ERR_TIMEOUT = 4      /* reserved: no call waits on the host          */
} pldp_status;

typedef enum { PLDP_F32 = 0, PLDP_BF16 = 1 } pldp_dtype;

typedef enum { PLDP_AGG_MAX = 0, PLDP_AGG_SUM = 1 } pldp_agg;

/* Per-sequence device status bits. */
#define PLDP_ST_CAND_OVERFLOW 1u  /* |P| > C_cap: the first C_cap positions are listed   */
#define PLDP_ST_TOKEN_RANGE   2u  /* a draft token outside [0, V)                        */
#define PLDP_ST_CAPACITY      4u  /* the append would pass T_cap: nothing appended       */
#define PLDP_ST_SEQ_LEN       8u  /* seq_len outside its valid range: sequence skipped   */
#define PLDP_ST_DRAFT_LEN    16u  /* draft_len outside [0, K]: clamped into it           */
#define PLDP_ST_ROW_INDEX    32u  /* a row_idx entry outside [0, R): that row ignored    */
#define PLDP_ST_TIMEOUT      64u  /* an on-chip copy did not complete in time: no result */

#define PLDP_MAX_NGRAM 8          /* largest ngram_max accepted                          */

/*
 * Candidate search -- Eq. 1 (Sec. 4.2):  P = { j | x_j = x_t, j < t },
 * narrowed by the longest-suffix n-gram rule of prompt lookup (Sec. 2, Fig. 2
 * caption): for n = ngram_max down to ngram_min, the first non-empty
 *   P_n = { j < t : j-n+1 >= 0 and x_{j-k} = x_{t-k} for k = 0..n-1 }
 * is P and n is match_len[b].  ngram_min = ngram_max = 1 is Eq. 1 itself.
 *
 *  ids        int32 [B, ids_stride]; row b holds the context of sequence b.
 *  ids_stride elements between rows (>= T_cap).
 *  seq_len    int32 [B]; valid range [0, T_cap] (else SEQ_LEN, nothing found).
 *  T_cap      row capacity: positions >= T_cap are never read.
 *  ngram_min, ngram_max   1 <= ngram_min <= ngram_max <= PLDP_MAX_NGRAM.
 *  cand_pos   int32 [B, C_cap] out: P in ascending order; slots past
 *             min(|P|, C_cap) are left untouched.
 *  C_cap      >= 0.  |P| > C_cap lists the first C_cap and sets CAND_OVERFLOW.
 *  cand_count int32 [B] out: the true |P| (even when it exceeds C_cap).
 *  match_len  int32 [B] out: the n of P, 0 when P is empty.
 *  status     uint32 [B] or NULL.
 * Fast path when ids is 16-byte aligned and ids_stride % 4 == 0.
 */
PLDP_API pldp_status pldp_find_candidates(const int32_t* ids, int64_t ids_stride,
                                          const int32_t* seq_len, int B, int64_t T_cap,
                                          int ngram_min, int ngram_max,
                                          int32_t* cand_pos, int C_cap,
                                          int32_t* cand_count, int32_t* match_len,
                                          uint32_t* status, void* stream);

/*
 * Ranking by hidden states -- Eq. 3 (Sec. 4.2.2):
 *   score_j = cos(H_{j-1}, H_{t-1}),  j* = argmax_{j in P} score_j,
 * with the optional threshold of App. B.3 (j kept only if score_j > threshold;
 * pass -INFINITY for none).  The caller passes the chosen layer l only.
 *
 *  H          [B, seq_stride] elements of dtype; row p of sequence b is
 *             H + b*seq_stride + p*d (rows are contiguous, d elements each).
 *  d          hidden width, 1 <= d and d * sizeof(dtype) <= 196608.
 *  seq_stride elements between sequences (>= T_cap * d).
 *  seq_len    int32 [B]; valid range [0, T_cap] (else SEQ_LEN, no result).
 *  T_cap      row capacity of H: rows >= T_cap are never read.
 *  cand_pos, cand_count, C_cap   as written by pldp_find_candidates; entries
 *             past min(cand_count, C_cap) are ignored.
 *  scores     float [B, C_cap] out or NULL: score of the i-th listed candidate.
 *             j = 0 (no H_{-1}) and positions outside [0, t) score -INFINITY
 *             and are never chosen.  A zero-norm row gives score 0.
 *  best_pos   int32 [B] out: j*, or -1 when no candidate is eligible.
 *  best_score float [B] out or NULL: score of j* (-INFINITY when none).
 *  status     uint32 [B] or NULL.
 * Scores are accumulated in fp32.  Ties go to the smaller position j; the
 * choice is deterministic for given inputs.  When H rows are 16-byte aligned
 * (H aligned, d*sizeof(dtype) and seq_stride*sizeof(dtype) multiples of 16)
 * the query row is staged in shared memory by a bulk asynchronous copy.
 */
PLDP_API pldp_status pldp_rank_hidden(const void* H, pldp_dtype dtype, int64_t d,
                                      int64_t seq_stride, const int32_t* seq_len, int B,
                                      int64_t T_cap, const int32_t* cand_pos,
                                      const int32_t* cand_count, int C_cap, float threshold,
                                      float* scores, int32_t* best_pos, float* best_score,
                                      uint32_t* status, void* stream);

/*
 * Ranking by averaged hidden states -- the variant of Eq. 3 studied in App. B.2
 * (the paper reports it does not help; it is here for completeness):
 *   Hbar_p  = mean(H_{max(0, p-m+1)}, ..., H_p)     (the m rows ending at p)
 *   score_j = cos(Hbar_{j-1}, Hbar_{t-1}),  j* = argmax_{j in P} score_j.
 * The printed formula averages H_1..H_m for every position; it is read as the
 * window of the m positions ending at the one averaged, cut at position 0.
 * m = 1 is Eq. 3.  Arguments, outputs and conventions as pldp_rank_hidden, plus
 *  m   window length, >= 1.
 * Limit: d * 4 <= 196608 (the query's window sum is held in fp32 in shared memory).
 */
PLDP_API pldp_status pldp_rank_hidden_avg(const void* H, pldp_dtype dtype, int64_t d,
                                          int64_t seq_stride, int m, const int32_t* seq_len, int B,
                                          int64_t T_cap, const int32_t* cand_pos,
                                          const int32_t* cand_count, int C_cap, float threshold,
                                          float* scores, int32_t* best_pos, float* best_score,
                                          uint32_t* status, void* stream);

/*
 * Ranking by attentions -- Eq. 2 (Sec. 4.2.1):
 *   score_j = max over the selected (layer, head) rows of A^{(l,g)}_{t-1}[j],
 *   j* = argmax_{j in P} score_j;  agg = PLDP_AGG_SUM sums the rows instead
 *   (the aggregation variant of Sec. 7.1).
 * The key index of Eq. 2 is read as the candidate j itself (the position an
 * induction head at query t-1 attends to is the token it copies).
 *
 *  A          dtype; for sequence b and row r the attention probabilities of
 *             query t-1 over keys:
 *               A + b*seq_stride + r*row_stride + key*key_stride.
 *             Rows with contiguous keys (key_stride = 1, row_stride >= T_cap) are
 *             the natural layout of one head's probabilities; the key-major layout
 *             (row_stride = 1, key_stride >= R) puts the R values of one key side
 *             by side, so each candidate's values are one contiguous read instead
 *             of R scattered 32-byte sectors.  A may also be page-locked host
 *             memory that device code can address (a cudaHostAlloc allocation
 *             under unified addressing): the kernels read only the selected rows'
 *             values at the candidate keys, so rows kept on the host need not be
 *             copied to the device whole.
 *  R          rows per sequence (>= 1).
 *  row_stride, key_stride   >= 1 (key_stride 0 is read as 1); the rows must not
 *             overlap: row_stride >= T_cap * key_stride or key_stride >= R *
 *             row_stride.  seq_stride >= (R-1)*row_stride + (T_cap-1)*key_stride + 1.
 *  row_idx    int32 [n_sel] device, or NULL for all R rows: the selected
 *             (layer, head) rows L* x G*.  Entries outside [0, R) are ignored
 *             and set ROW_INDEX.
 *  seq_len, T_cap, cand_pos, cand_count, C_cap, status   as pldp_rank_hidden.
 *  scores     float [B, C_cap] out or NULL.  Positions outside [0, t) score
 *             -INFINITY and are never chosen.
 *  best_pos, best_score   as pldp_rank_hidden.  Ties go to the smaller j.
 * MAX is exact; SUM accumulates in fp32 in a fixed order.
 */
PLDP_API pldp_status pldp_rank_attention(const void* A, pldp_dtype dtype, int R,
                                         int64_t row_stride, int64_t key_stride, int64_t seq_stride,
                                         const int32_t* row_idx, int n_sel, pldp_agg agg,
                                         const int32_t* seq_len, int B, int64_t T_cap,
                                         const int32_t* cand_pos, const int32_t* cand_count,
                                         int C_cap, float* scores, int32_t* best_pos,
                                         float* best_score, uint32_t* status, void* stream);

/*
 * Draft prediction -- Sec. 4.3:  xhat_i = x_{j*+i}, i = 1..K.
 * The span stops at the last token x_t: draft_len[b] = min(K, t - j*) tokens,
 * the rest of draft[b, :] is -1.  best_pos[b] = -1 (or outside [0, t), or an
 * invalid seq_len) gives draft_len 0.
 *
 *  ids, ids_stride, seq_len, T_cap   as pldp_find_candidates.
 *  best_pos   int32 [B].
 *  K          draft length, >= 1.
 *  draft      int32 [B, K] out;  draft_len  int32 [B] out.
 */
PLDP_API pldp_status pldp_extract_draft(const int32_t* ids, int64_t ids_stride,
                                        const int32_t* seq_len, int64_t T_cap,
                                        const int32_t* best_pos, int B, int K,
                                        int32_t* draft, int32_t* draft_len, void* stream);

/*
 * The drafting half of a step in one call: candidate search, ranking by hidden
 * states and/or attentions, and draft extraction, with the results of
 * pldp_find_candidates, pldp_rank_hidden, pldp_rank_attention and
 * pldp_extract_draft called in turn (same conventions, same status bits; the
 * fp32 score sums may be split differently, so scores can differ in the last
 * bits and a tie within rounding may be broken differently).  Eq. 1-3
 * (Sec. 4.2) and Sec. 4.3.
 *
 * One launch over a flat (chunk, sequence) grid.  Each CTA streams its chunk of
 * the context, scores every occurrence of x_t it finds (cosine and attention
 * score, with all its threads) and records it with its suffix-match length in a
 * small per-sequence list held in the workspace; the CTA that finishes a
 * sequence last (an atomic ticket, no waiting) orders the list into the
 * candidate list, picks the best of each ranking and writes the draft.  More
 * than 256 occurrences in a sequence fall back to an ordered rescan of its
 * context by that CTA.
 *
 * Fields of the argument block (device pointers unless stated):
 *  ids .. match_len      as pldp_find_candidates (T_cap <= 2^27).
 *  H .. best_h_score     as pldp_rank_hidden (H = NULL skips hidden ranking;
 *                        H rows must be 16-byte aligned).  h_scores and
 *                        best_h_score may be NULL.
 *  A .. best_a_score     as pldp_rank_attention (A = NULL skips it; either
 *                        layout, a_key_stride as its key_stride; A may be
 *                        device-addressable page-locked host memory); a_scores
 *                        and best_a_score may be NULL.
 *  draft_from            0: draft after best_h, 1: after best_a (that ranking
 *                        must be given).
 *  K, draft, draft_len   as pldp_extract_draft.
 *  status                uint32 [B] or NULL.
 *  workspace             device scratch of pldp_draft_workspace_size(B) bytes,
 *                        16-byte aligned, ZEROED by the caller before its first
 *                        use; every call leaves it zeroed again.  Calls that may
 *                        run concurrently need separate workspaces.  May be NULL
 *                        when an index is given.
 *  index, index_bytes, V optional incremental token index (NULL: scan the
 *                        contexts): device memory of pldp_index_size(B, V)
 *                        bytes, built by pldp_index_build, for token ids in
 *                        [0, V).  With it, a step looks up the occurrences of
 *                        x_t instead of scanning the context, and appends the
 *                        positions added since the last step; results are the
 *                        same as without it (a token with more than 15 earlier
 *                        occurrences, or a sequence whose index is unusable,
 *                        is scanned).  The index must only ever see the
 *                        contexts grow by appending: a sequence whose length
 *                        fell below what was indexed is marked unusable (and
 *                        scanned) until the index is rebuilt.
 * Layouts the fused path does not take return PLDP_ERR_UNSUPPORTED; the
 * separate calls accept them.
 */
typedef struct pldp_draft_step_args {
    const int32_t* ids;
    int64_t ids_stride;
    const int32_t* seq_len;
    int B;
    int64_t T_cap;
    int ngram_min;
    int ngram_max;
    int32_t* cand_pos;
    int C_cap;
    int32_t* cand_count;
    int32_t* match_len;
    const void* H;
    pldp_dtype h_dtype;
    int64_t d;
    int64_t h_seq_stride;
    float threshold;
    float* h_scores;
    int32_t* best_h;
    float* best_h_score;
    const void* A;
    pldp_dtype a_dtype;
    int R;
    int64_t a_row_stride;
    int64_t a_key_stride;   /* elements between keys of a row; 0 is read as 1 */
    int64_t a_seq_stride;
    const int32_t* row_idx;
    int n_sel;
    pldp_agg agg;
    float* a_scores;
    int32_t* best_a;
    float* best_a_score;
    int draft_from;
    int K;
    int32_t* draft;
    int32_t* draft_len;
    uint32_t* status;
    void* workspace;
    size_t workspace_bytes;
    void* index;
    size_t index_bytes;
    int V;
} pldp_draft_step_args;

/* `args` is a HOST pointer to the argument block, read before the call returns. */
PLDP_API pldp_status pldp_draft_step(const pldp_draft_step_args* args, void* stream);

/* Bytes of workspace pldp_draft_step needs for B sequences (0 if B < 0). */
PLDP_API size_t pldp_draft_workspace_size(int B);

/*
 * The incremental token index of pldp_draft_step (no counterpart in the paper:
 * it is a way to find the occurrences of Eq. 1 without rescanning the context).
 * Per sequence and token it holds the number of occurrences among the indexed
 * positions and up to 15 of them (one 64-byte entry); per sequence the number of
 * positions indexed.
 * pldp_index_build clears `index` and indexes positions 0 .. seq_len[b]-2 of
 * every sequence (all but the last token, which the next draft step looks up).
 * Token ids outside [0, V) mark that sequence's index unusable (TOKEN_RANGE);
 * seq_len outside [0, T_cap] too (SEQ_LEN).  Memory: about B * V * 64 bytes.
 */
PLDP_API size_t pldp_index_size(int B, int V);
PLDP_API pldp_status pldp_index_build(const int32_t* ids, int64_t ids_stride, const int32_t* seq_len,
                                      int B, int64_t T_cap, int V, void* index,
                                      size_t index_bytes, uint32_t* status, void* stream);

/*
 * Greedy verification -- Sec. 4.4 at temperature 0, with the K+1 next-token
 * distributions of one forward pass on the draft (Sec. 3):
 *   a_i   = argmax_v logits[b, i, v], i = 0..K   (smallest v among equal maxima;
 *           -0.0 equals +0.0)
 *   n     = first i < draft_len[b] with draft[b, i] != a_i, else draft_len[b]
 *   bonus = a_n
 * accept_len[b] = n and next_token[b] = bonus: the step emits
 * draft[b, 0..n-1] followed by bonus, exactly what greedy decoding emits.
 *
 *  logits     dtype [B, K+1, V], contiguous.  Fast path when logits is 16-byte
 *             aligned and V * sizeof(dtype) is a multiple of 16.
 *  draft      int32 [B, K];  draft_len  int32 [B] (outside [0, K]: clamped,
 *             DRAFT_LEN).  Draft tokens outside [0, V) never match (TOKEN_RANGE).
 *  argmax     int32 [B, K+1] out or NULL: every a_i.
 *  accept_len int32 [B] out;  next_token int32 [B] out.
 *  seq_len    int32 [B] in/out or NULL.  When given (valid range [1, T_cap],
 *             else SEQ_LEN and no bookkeeping for b), with L the old value:
 *               kv_keep_len[b] = L + n   (x_t and the n accepted tokens are the
 *                                         positions whose keys/values survive)
 *               if L + n + 1 <= T_cap: ids[b, L..L+n-1] = draft[b, 0..n-1],
 *                 ids[b, L+n] = bonus (ids may be NULL), seq_len[b] = L + n + 1;
 *               else CAPACITY and neither ids nor seq_len changes.
 *  ids, ids_stride, T_cap   the context rows to append to (ids may be NULL).
 *  kv_keep_len int32 [B] out or NULL (needs seq_len).
 *  status     uint32 [B] or NULL.
 *  workspace  device scratch of at least pldp_verify_workspace_size(B, K, V)
 *             bytes, 16-byte aligned, ZEROED by the caller before its first
 *             use.  Every call returns it to all-zero when it completes, so
 *             it can be reused by the next call on the same stream (or graph
 *             replay) without clearing.  Calls that may run concurrently need
 *             separate workspaces.
 */
PLDP_API pldp_status pldp_verify_greedy(const void* logits, pldp_dtype dtype, int B, int K,
                                        int V, const int32_t* draft, const int32_t* draft_len,
                                        int32_t* argmax, int32_t* accept_len,
                                        int32_t* next_token, int32_t* ids, int64_t ids_stride,
                                        int32_t* seq_len, int64_t T_cap, int32_t* kv_keep_len,
                                        uint32_t* status, void* workspace,
                                        size_t workspace_bytes, void* stream);

/*
 * Greedy verification of the current step followed by the drafting of the next
 * one, in one call -- pldp_verify_greedy then pldp_draft_step (with the token
 * index) on the context it has just extended, with the same results and status
 * bits as those two calls in turn.  The paper has no counterpart: in a decode
 * loop the next draft depends only on this step's verification (the accepted
 * tokens, the bonus token) and on the hidden states and attention rows of the
 * forward pass that produced this step's logits, so nothing runs between the
 * two.  The argmax pass is followed, one CTA per sequence, by the accept/bonus/
 * append of verification and then the candidate search, ranking and draft of
 * the next step.
 *
 *  logits, dtype, V   this step's logits [B, K+1, V], as pldp_verify_greedy.
 *  draft, draft_len   this step's draft [B, K] and lengths [B]; they may be the
 *                     same buffers as next.draft and next.draft_len (each
 *                     sequence's draft is read before it is replaced).
 *  argmax, accept_len, next_token, kv_keep_len, workspace, workspace_bytes
 *                     as pldp_verify_greedy (workspace zeroed before first use;
 *                     every call leaves it zero).
 *  next               the next step's pldp_draft_step arguments.  next.index is
 *                     required (built by pldp_index_build, with next.V == V).
 *                     next.B and next.K are the verification's B and K;
 *                     next.ids, next.ids_stride, next.seq_len and next.T_cap are
 *                     the context verification appends to (read and WRITTEN by
 *                     this call); next.status receives both calls' bits.
 *                     next.workspace is not used.
 */
typedef struct pldp_verify_draft_args {
    const void* logits;
    pldp_dtype dtype;
    int V;
    const int32_t* draft;
    const int32_t* draft_len;
    int32_t* argmax;
    int32_t* accept_len;
    int32_t* next_token;
    int32_t* kv_keep_len;
    void* workspace;
    size_t workspace_bytes;
    pldp_draft_step_args next;
} pldp_verify_draft_args;

/* `args` is a HOST pointer to the argument block, read before the call returns. */
PLDP_API pldp_status pldp_verify_greedy_draft(const pldp_verify_draft_args* args, void* stream);

/*
 * Sampling verification -- Sec. 4.4 at temperature T > 0 (the paper's sampled
 * runs use T = 1, Table 2).  Position i of sequence b draws
 *   y_i = the smallest v with sum_{v' <= v} p_v' > u[b, i],
 *         p = softmax(logits[b, i] / T)                  (inverse-CDF sampling)
 * from the caller's uniform u[b, i]; then, as for greedy verification,
 *   n = first i < draft_len[b] with draft[b, i] != y_i, else draft_len[b];
 *   bonus = y_n.
 * For a draft with one token per position (PLD+'s draft) this accepts draft_i
 * with probability p(draft_i) and on a rejection draws the bonus from p
 * restricted to the other tokens: the step emits exactly what sampling from the
 * target alone would.  The random numbers are inputs: the same uniforms give
 * the same draws.
 *
 *  logits        dtype [B, K+1, V], contiguous, finite.  Fast path when logits is
 *                16-byte aligned and V * sizeof(dtype) is a multiple of 16.
 *  temperature   T > 0, finite (else PLDP_ERR_INVALID_ARG).
 *  uniforms      float [B, K+1]; values outside [0, 1) are clamped into it.
 *  sampled       int32 [B, K+1] out or NULL: every y_i.
 *  draft, draft_len, accept_len, next_token, ids, ids_stride, seq_len, T_cap,
 *  kv_keep_len, status   as pldp_verify_greedy.
 *  workspace     device scratch of pldp_verify_sample_workspace_size(B, K, V, dtype)
 *                bytes, 16-byte aligned (no zeroing needed).
 * Probabilities are computed in fp32 (per-2 KB-piece maxima and sums of
 * exp2(log2(e) (l - max) / T)); a draw can differ from the exact draw only when
 * u lies within fp32 rounding (~1e-6) of a boundary of the cumulative
 * distribution.  K + 1 <= 12288.
 */
PLDP_API pldp_status pldp_verify_sample(const void* logits, pldp_dtype dtype, int B, int K, int V,
                                        float temperature, const float* uniforms,
                                        const int32_t* draft, const int32_t* draft_len,
                                        int32_t* sampled, int32_t* accept_len,
                                        int32_t* next_token, int32_t* ids, int64_t ids_stride,
                                        int32_t* seq_len, int64_t T_cap, int32_t* kv_keep_len,
                                        uint32_t* status, void* workspace,
                                        size_t workspace_bytes, void* stream);

/* Bytes of workspace pldp_verify_sample needs (0 if invalid). */
PLDP_API size_t pldp_verify_sample_workspace_size(int B, int K, int V, pldp_dtype dtype);

/*
 * Sampling verification of the current step followed by the drafting of the
 * next one, in one call -- pldp_verify_sample then pldp_draft_step (with the
 * token index) on the context it has just extended, with the same results and
 * status bits as those two calls in turn.  Sec. 4.4 at temperature T > 0 (the
 * paper's sampled runs use T = 1, Table 2), then Eq. 1-3 and Sec. 4.3; the paper
 * has no fused form.  Three launches: the per-piece stats pass over the logits,
 * one warp per row that draws, then one CTA per sequence that accepts, appends
 * and drafts the next step.
 *
 *  logits, dtype, V   this step's logits [B, K+1, V], as pldp_verify_sample.
 *  temperature        T > 0, finite (else PLDP_ERR_INVALID_ARG).
 *  uniforms           float [B, K+1], as pldp_verify_sample (clamped into [0, 1)).
 *  draft, draft_len   this step's draft [B, K] and lengths [B]; they may be the
 *                     same buffers as next.draft and next.draft_len.
 *  sampled            int32 [B, K+1] out or NULL: every draw y_i.
 *  accept_len, next_token, kv_keep_len   as pldp_verify_greedy.
 *  workspace          device scratch of pldp_verify_sample_draft_workspace_size(
 *                     B, K, V, dtype) bytes, 16-byte aligned (no zeroing needed).
 *                     Calls that may run concurrently need separate workspaces.
 *  next               the next step's pldp_draft_step arguments, as for
 *                     pldp_verify_greedy_draft (next.index required, next.V == V,
 *                     next.B and next.K are the verification's B and K, next.ids /
 *                     next.seq_len are appended to, next.status receives both
 *                     calls' bits, next.workspace is not used).
 * K + 1 <= 12288.  The draws are those of pldp_verify_sample on the same inputs.
 */
typedef struct pldp_verify_sample_draft_args {
    const void* logits;
    pldp_dtype dtype;
    int V;
    float temperature;
    const float* uniforms;
    const int32_t* draft;
    const int32_t* draft_len;
    int32_t* sampled;
    int32_t* accept_len;
    int32_t* next_token;
    int32_t* kv_keep_len;
    void* workspace;
    size_t workspace_bytes;
    pldp_draft_step_args next;
} pldp_verify_sample_draft_args;

/* `args` is a HOST pointer to the argument block, read before the call returns. */
PLDP_API pldp_status pldp_verify_sample_draft(const pldp_verify_sample_draft_args* args, void* stream);

/* Bytes of workspace pldp_verify_sample_draft needs (0 if invalid). */
PLDP_API size_t pldp_verify_sample_draft_workspace_size(int B, int K, int V, pldp_dtype dtype);

/*
 * Greedy verification without a caller workspace.  The paper has no counterpart:
 * this is a deployment convenience.  Same arguments, results and status bits as
 * pldp_verify_greedy, minus the workspace.
 *
 * Who needs it: callers that cannot allocate device memory for a workspace --
 * code embedded in a host program that owns every GPU allocation, and serving
 * loops that must not call cudaMalloc/cudaFree after start-up because those
 * calls can synchronise the whole device.
 *
 * The scratch lives in a fixed 1 MiB area compiled into the library; every GPU
 * that loads the library keeps it until the process exits.  Requests needing
 * more than that (pldp_verify_workspace_size(B, K, V) > 1048576, i.e. roughly
 * B*(K+1) > 130000 rows) are rejected with PLDP_ERR_INVALID_ARG.  The call
 * allocates nothing: it clears the part of the area it uses with
 * cudaMemsetAsync on `stream`, then launches the verification kernels.
 *
 * Every call looks up the area's device address in the CUDA context current on
 * the calling thread (cudaGetSymbolAddress, which allocates nothing), so a
 * switch of context or a device reset between calls never leaves it a stale
 * address.  The first call in a context also makes the runtime load the
 * library's device code there; make that first call before any stream capture.
 * All calls on a device share the one area, which keeps whatever the last call
 * left there: calls that can overlap on the GPU (different streams, or threads
 * without ordering between them) race on it and must be serialised by the
 * caller.
 */
PLDP_API pldp_status pldp_verify_greedy_noalloc(const void* logits, pldp_dtype dtype, int B,
                                                int K, int V, const int32_t* draft,
                                                const int32_t* draft_len, int32_t* argmax,
                                                int32_t* accept_len, int32_t* next_token,
                                                int32_t* ids, int64_t ids_stride,
                                                int32_t* seq_len, int64_t T_cap,
                                                int32_t* kv_keep_len, uint32_t* status,
                                                void* stream);

/* Bytes of workspace pldp_verify_greedy needs for these sizes (0 if invalid). */
PLDP_API size_t pldp_verify_workspace_size(int B, int K, int V);

/*
 * Induction-head identification -- Sec. 4.2.1, the offline step that picks the
 * (layer, head) rows Eq. 2 aggregates.  Each observation b is a generated token
 * x_p (p = pos[b]) with its context ids[b, 0..p] and the attention rows of query
 * p-1 over keys 0..p-1 for R candidate (layer, head) rows:
 *   P      = {j < p : x_j = x_p}
 *   ov(j)  = the largest k <= max_suffix with x_{j-i} = x_{p-i} for all i < k
 *   r*     = argmax_{j in P} ov(j)              (the smaller j on ties)
 *   counts[r] += 1 when row r's largest attention is at key r*
 *                                               (the smaller key on ties)
 * The paper's rule is read per row: a head counts when r* is where its own
 * attention peaks.  Run it over many observations, then keep the rows with the
 * most counts (pldp_top_heads).
 *
 *  B          observations, at most 65535 (else PLDP_ERR_UNSUPPORTED).
 *  ids, ids_stride, T_cap   int32 contexts [B, ids_stride], T_cap <= ids_stride.
 *  pos        int32 [B]; outside [1, T_cap - 1]: SEQ_LEN, nothing counted.
 *  max_suffix >= 1: cap on ov(j).
 *  A          dtype [B, seq_stride]: row r of observation b at
 *             A + b*seq_stride + r*row_stride, keys 0..p-1 (row_stride >= T_cap,
 *             seq_stride >= R*row_stride).
 *  counts     uint32 [R], ADDED to (initialise once, accumulate over calls).
 *  r_star     int32 [B] out or NULL: r*, -1 when x_p does not occur before p.
 *  status     uint32 [B] or NULL.
 * Atomic adds on counts: concurrent calls on one counts array accumulate
 * correctly.  Offline utility: not part of the decode step.
 */
PLDP_API pldp_status pldp_identify_heads(const int32_t* ids, int64_t ids_stride, const int32_t* pos,
                                         int B, int64_t T_cap, int max_suffix, const void* A,
                                         pldp_dtype dtype, int R, int64_t row_stride,
                                         int64_t seq_stride, uint32_t* counts, int32_t* r_star,
                                         uint32_t* status, void* stream);

/*
 * The k rows with the most counts (ties to the smaller row index), written in
 * that order to row_idx int32 [k] -- the row_idx argument of pldp_rank_attention.
 * 1 <= k <= R <= 8192.  counts: uint32 [R] (device).
 */
PLDP_API pldp_status pldp_top_heads(const uint32_t* counts, int R, int k, int32_t* row_idx, void* stream);

/* Message describing the last failed call on this host thread ("" if none). */
PLDP_API const char* pldp_last_error(void);

/* Library version (major * 10000 + minor * 100 + patch). */
PLDP_API int pldp_version(void);

#ifdef __cplusplus
}
#endif

#endif /* PLDP_H */
