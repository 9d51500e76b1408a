// pldp_draft_step: the drafting half of a PLD+ step in one kernel -- candidate
// search (Eq. 1 with the longest-suffix n-gram rule), ranking by hidden states
// (Eq. 3) and/or by attentions (Eq. 2), and draft extraction (Sec. 4.3).
//
// One thread-block cluster per sequence.  Every CTA scans a chunk of the
// context; counts meet over distributed shared memory and the matches are
// written in order (pldp_scan.cuh).  The CTAs then split the ranking: with two
// or more CTAs, the even ranks score hidden states while the odd ranks score
// attentions, in parallel.  The query row H_{t-1} depends only on seq_len, so
// its bulk asynchronous copy into shared memory is issued at kernel entry and
// lands while the scan streams.  CTA 0 combines the CTAs' best keys and writes
// the draft.  The results are those of pldp_find_candidates, pldp_rank_hidden,
// pldp_rank_attention and pldp_extract_draft called in turn (fp32 score sums
// may be split differently, so scores can differ in their last bits).
#include <type_traits>

#include "pldp_rank.cuh"
#include "pldp_scan.cuh"

namespace pldp {
namespace {

constexpr int kThreads = 256;
constexpr int64_t kPositionsPerCta = 4096;
constexpr size_t kMaxQueryBytes = 196608;
constexpr int kMaxSelRows = 8192;

struct NoHidden {};

struct DraftParams {
    const int32_t* ids;
    int64_t ids_stride;
    const int32_t* seq_len;
    int64_t T_cap;
    int ngram_min, ngram_max;
    int32_t* cand_pos;
    int C_cap;
    int32_t* cand_count;
    int32_t* match_len;
    const void* H;
    int64_t d;
    int64_t h_seq_stride;
    float threshold;
    float* h_scores;
    int32_t* best_h;
    float* best_h_score;
    const void* A;
    bool a_bf16;
    int R;
    int64_t a_row_stride;
    int64_t a_seq_stride;
    const int32_t* row_idx;
    int n_sel;
    int agg;
    float* a_scores;
    int32_t* best_a;
    float* best_a_score;
    int draft_from;   // 0: hidden choice, 1: attention choice
    int K;
    int32_t* draft;
    int32_t* draft_len;
    uint32_t* status;
    int64_t chunk;
    size_t rows_offset;   // byte offset of the attention row table in dynamic shared memory
};

struct CtaBest {
    unsigned long long hkey, akey;
    int err;
};

template <typename TH>
__global__ void __launch_bounds__(kThreads) draft_step_kernel(const DraftParams p) {
    constexpr bool HAS_H = !std::is_same<TH, NoHidden>::value;
    using TQ = typename std::conditional<HAS_H, TH, float>::type;
    extern __shared__ __align__(128) unsigned char dyn_smem[];
    TQ* q_sh = reinterpret_cast<TQ*>(dyn_smem);                                // H_{t-1}
    int64_t* rows_sh = reinterpret_cast<int64_t*>(dyn_smem + p.rows_offset);   // attention rows
    __shared__ ScanShared ss;
    __shared__ RankShared hs, as;
    __shared__ CtaBest mine;
    __shared__ __align__(8) uint64_t bar;
    __shared__ int bad_rows;

    cg::cluster_group cluster = cg::this_cluster();
    const int CL = static_cast<int>(cluster.num_blocks());
    const int rank = static_cast<int>(cluster.block_rank());
    const int b = blockIdx.x / CL;
    const int tid = threadIdx.x;
    const bool has_a = p.A != nullptr;

    const int64_t L = p.seq_len[b];
    if (L < 0 || L > p.T_cap) {       // cluster-uniform exit: nothing to draft
        if (rank == 0) {
            for (int i = tid; i < p.K; i += kThreads) p.draft[static_cast<int64_t>(b) * p.K + i] = -1;
            if (tid == 0) {
                p.cand_count[b] = 0;
                p.match_len[b] = 0;
                if (HAS_H) {
                    p.best_h[b] = -1;
                    if (p.best_h_score) p.best_h_score[b] = -INFINITY;
                }
                if (has_a) {
                    p.best_a[b] = -1;
                    if (p.best_a_score) p.best_a_score[b] = -INFINITY;
                }
                p.draft_len[b] = 0;
                if (p.status) atomicOr(p.status + b, PLDP_ST_SEQ_LEN);
            }
        }
        return;
    }
    const int64_t t = L - 1;
    const bool hidden_team = HAS_H && (CL == 1 || (rank & 1) == 0);
    const bool attn_team = has_a && (CL == 1 || (rank & 1) == 1);
    const int h_S = CL == 1 ? 1 : (CL + 1) / 2, a_S = CL == 1 ? 1 : CL / 2;
    const int team_rank = CL == 1 ? 0 : rank / 2;

    // Query row: needed as soon as any candidate is, and known from seq_len alone.
    const bool q_fetch = hidden_team && t >= 2;
    const TQ* hb = nullptr;
    if constexpr (HAS_H) hb = static_cast<const TQ*>(p.H) + static_cast<int64_t>(b) * p.h_seq_stride;
    if constexpr (HAS_H) {
        if (q_fetch && tid == 0) {
            const uint32_t qbytes = static_cast<uint32_t>(p.d * sizeof(TQ));
            mbar_init(&bar, 1);
            fence_mbar_init();
            mbar_arrive_expect_tx(&bar, qbytes);
            bulk_g2s(q_sh, hb + (t - 1) * p.d, qbytes, &bar);
        }
    }
    if (tid <= PLDP_MAX_NGRAM) ss.cnt[tid] = 0;
    rank_shared_init(hs);
    rank_shared_init(as);

    // ---- candidate search --------------------------------------------------------
    const int32_t* row = p.ids + static_cast<int64_t>(b) * p.ids_stride;
    const int64_t c0 = static_cast<int64_t>(rank) * p.chunk;
    const int64_t c1 = min(c0 + p.chunk, t);
    int c[PLDP_MAX_NGRAM];
#pragma unroll
    for (int k = 0; k < PLDP_MAX_NGRAM; ++k) c[k] = 0;
    if (t >= 1) scan_count<true>(row, c0, c1, t, p.ngram_max, c);
    __syncthreads();
    scan_reduce_counts(c, p.ngram_max, ss);
    cluster.sync();                                     // (1) all counts final
    scan_decide(cluster, ss, CL, rank, p.ngram_min, p.ngram_max);
    if (rank == 0 && tid == 0) {
        p.cand_count[b] = ss.total;
        p.match_len[b] = ss.nstar;
        if (p.status && ss.total > p.C_cap) atomicOr(p.status + b, PLDP_ST_CAND_OVERFLOW);
    }
    int32_t* cand_row = p.cand_pos + static_cast<int64_t>(b) * p.C_cap;
    scan_write<true>(row, c0, c1, t, p.ngram_max, ss, cand_row, p.C_cap);
    bool bad = false;
    if (attn_team) bad = stage_rows(rows_sh, p.row_idx, p.n_sel, p.R, p.a_row_stride, &bad_rows);
    cluster.sync();                                     // (2) the candidate list is complete
    const int n = ss.total < p.C_cap ? ss.total : p.C_cap;

    // ---- ranking -------------------------------------------------------------------
    if constexpr (HAS_H) {
        if (hidden_team)
            hidden_rank_cta<TQ, true>(hb, p.d, t, cand_row, n, h_S, team_rank, nullptr, q_sh, &bar,
                                      q_fetch, p.threshold,
                                      p.h_scores ? p.h_scores + static_cast<int64_t>(b) * p.C_cap : nullptr,
                                      hs);
        // the copy into this CTA's shared memory must have landed before exit (bounded)
        if (q_fetch && tid == 0 && !mbar_wait(&bar, 0, kMbarPolls)) hs.err = 1;
    }
    if (attn_team) {
        if (bad && team_rank == 0 && tid == 0 && p.status) atomicOr(p.status + b, PLDP_ST_ROW_INDEX);
        const size_t es = p.a_bf16 ? 2 : 4;
        const void* ab = static_cast<const char*>(p.A) + static_cast<int64_t>(b) * p.a_seq_stride * es;
        attention_rank_cta(ab, p.a_bf16, rows_sh, p.n_sel, t, cand_row, n, a_S, team_rank, nullptr,
                           p.agg == PLDP_AGG_MAX,
                           p.a_scores ? p.a_scores + static_cast<int64_t>(b) * p.C_cap : nullptr, as);
    }
    __syncthreads();
    if (tid == 0) {
        mine.hkey = rank_best_key(hs);
        mine.akey = rank_best_key(as);
        mine.err = hs.err;
    }
    cluster.sync();                                     // (3) every CTA's best is final

    // ---- combine and draft (CTA 0, warp 0) ------------------------------------------
    if (rank == 0 && tid < 32) {
        unsigned long long hk = 0, ak = 0;
        int err = 0;
        if (tid < CL) {
            const CtaBest* remote = cluster.map_shared_rank(&mine, tid);
            hk = remote->hkey;
            ak = remote->akey;
            err = remote->err;
        }
        hk = warp_max_u64(hk);
        ak = warp_max_u64(ak);
        err = static_cast<int>(__reduce_or_sync(0xFFFFFFFFu, static_cast<unsigned>(err)));
        const int32_t bh = (err || hk == 0) ? -1 : static_cast<int32_t>(key_index(hk));
        const int32_t ba = ak == 0 ? -1 : static_cast<int32_t>(key_index(ak));
        if (tid == 0) {
            if (HAS_H) {
                p.best_h[b] = bh;
                if (p.best_h_score) p.best_h_score[b] = bh >= 0 ? key_value(hk) : -INFINITY;
                if (err && p.status) atomicOr(p.status + b, PLDP_ST_TIMEOUT);
            }
            if (has_a) {
                p.best_a[b] = ba;
                if (p.best_a_score) p.best_a_score[b] = ba >= 0 ? key_value(ak) : -INFINITY;
            }
        }
        const int64_t js = p.draft_from == 0 ? bh : ba;
        int64_t dl = 0;
        if (js >= 0 && js < t) dl = (t - js < p.K) ? (t - js) : p.K;
        for (int i = tid; i < p.K; i += 32)
            p.draft[static_cast<int64_t>(b) * p.K + i] = (i < dl) ? __ldg(row + js + 1 + i) : -1;
        if (tid == 0) p.draft_len[b] = static_cast<int32_t>(dl);
    }
    cluster_arrive();
    cluster_wait();                                     // (4) CTA 0's remote reads are done
}

template <typename TH>
pldp_status launch_draft_step(DraftParams p, int B, size_t smem, cudaStream_t s) {
    const void* fn = reinterpret_cast<const void*>(&draft_step_kernel<TH>);
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(draft_step_kernel<TH>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess)
            return fail(PLDP_ERR_CUDA, "draft_step: shared memory attribute: %s", cudaGetErrorString(e));
    }
    int CL;
    scan_shape(p.T_cap, B, resident_blocks(fn, kThreads, smem), kPositionsPerCta, &CL, &p.chunk);
    if (static_cast<int64_t>(B) * CL > INT32_MAX) return fail(PLDP_ERR_INVALID_ARG, "draft_step: B too large");
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(B * CL));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CL;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, draft_step_kernel<TH>, p);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "draft_step: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}

}  // namespace
}  // namespace pldp

using namespace pldp;

extern "C" PLDP_API pldp_status pldp_draft_step(const pldp_draft_step_args* a, void* stream) {
    if (!a) return fail(PLDP_ERR_INVALID_ARG, "draft_step: null argument block");
    const int B = a->B;
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "draft_step: B < 0");
    if (a->T_cap < 0 || a->T_cap > INT32_MAX) return fail(PLDP_ERR_INVALID_ARG, "draft_step: bad T_cap");
    if (a->ids_stride < a->T_cap) return fail(PLDP_ERR_INVALID_ARG, "draft_step: ids_stride < T_cap");
    if (a->ngram_min < 1 || a->ngram_max < a->ngram_min || a->ngram_max > PLDP_MAX_NGRAM)
        return fail(PLDP_ERR_INVALID_ARG, "draft_step: need 1 <= ngram_min <= ngram_max <= %d",
                    PLDP_MAX_NGRAM);
    if (a->C_cap < 0) return fail(PLDP_ERR_INVALID_ARG, "draft_step: C_cap < 0");
    if (a->K < 1) return fail(PLDP_ERR_INVALID_ARG, "draft_step: K < 1");
    if (!a->H && !a->A) return fail(PLDP_ERR_INVALID_ARG, "draft_step: neither H nor A given");
    if (a->draft_from != 0 && a->draft_from != 1)
        return fail(PLDP_ERR_INVALID_ARG, "draft_step: draft_from must be 0 (hidden) or 1 (attention)");
    if ((a->draft_from == 0 && !a->H) || (a->draft_from == 1 && !a->A))
        return fail(PLDP_ERR_INVALID_ARG, "draft_step: draft_from names a ranking that is not given");
    size_t qbytes = 0, h_es = 0;
    if (a->H) {
        if (a->h_dtype != PLDP_F32 && a->h_dtype != PLDP_BF16)
            return fail(PLDP_ERR_UNSUPPORTED, "draft_step: unsupported hidden dtype %d", (int)a->h_dtype);
        h_es = a->h_dtype == PLDP_F32 ? 4 : 2;
        if (a->d < 1) return fail(PLDP_ERR_INVALID_ARG, "draft_step: d < 1");
        qbytes = static_cast<size_t>(a->d) * h_es;
        if (qbytes > kMaxQueryBytes)
            return fail(PLDP_ERR_UNSUPPORTED, "draft_step: d * sizeof(dtype) > %zu", kMaxQueryBytes);
        if (a->h_seq_stride < a->T_cap * a->d)
            return fail(PLDP_ERR_INVALID_ARG, "draft_step: h_seq_stride < T_cap*d");
        if (a->threshold != a->threshold) return fail(PLDP_ERR_INVALID_ARG, "draft_step: threshold is NaN");
    }
    int sel = 0;
    if (a->A) {
        if (a->a_dtype != PLDP_F32 && a->a_dtype != PLDP_BF16)
            return fail(PLDP_ERR_UNSUPPORTED, "draft_step: unsupported attention dtype %d", (int)a->a_dtype);
        if (a->agg != PLDP_AGG_MAX && a->agg != PLDP_AGG_SUM)
            return fail(PLDP_ERR_INVALID_ARG, "draft_step: unknown aggregation %d", (int)a->agg);
        if (a->R < 1) return fail(PLDP_ERR_INVALID_ARG, "draft_step: R < 1");
        if (a->a_row_stride < a->T_cap) return fail(PLDP_ERR_INVALID_ARG, "draft_step: a_row_stride < T_cap");
        if (a->a_seq_stride < static_cast<int64_t>(a->R) * a->a_row_stride)
            return fail(PLDP_ERR_INVALID_ARG, "draft_step: a_seq_stride < R*a_row_stride");
        sel = a->row_idx ? a->n_sel : a->R;
        if (sel < 1 || sel > kMaxSelRows)
            return fail(PLDP_ERR_INVALID_ARG, "draft_step: need 1 <= n_sel <= %d", kMaxSelRows);
    }
    if (B == 0) return PLDP_OK;
    if (!a->ids || !a->seq_len || !a->cand_count || !a->match_len || !a->draft || !a->draft_len ||
        (a->C_cap > 0 && !a->cand_pos) || (a->H && !a->best_h) || (a->A && !a->best_a))
        return fail(PLDP_ERR_INVALID_ARG, "draft_step: null pointer");
    if (!(aligned16(a->ids) && a->ids_stride % 4 == 0 && a->T_cap % 4 == 0))
        return fail(PLDP_ERR_UNSUPPORTED,
                    "draft_step: ids must be 16-byte aligned with ids_stride and T_cap multiples of 4 "
                    "(the separate calls accept any layout)");
    if (a->H && !(aligned16(a->H) && qbytes % 16 == 0 && (a->h_seq_stride * h_es) % 16 == 0))
        return fail(PLDP_ERR_UNSUPPORTED,
                    "draft_step: hidden rows must be 16-byte aligned (the separate calls accept any layout)");

    DraftParams p = {};
    p.ids = a->ids;
    p.ids_stride = a->ids_stride;
    p.seq_len = a->seq_len;
    p.T_cap = a->T_cap;
    p.ngram_min = a->ngram_min;
    p.ngram_max = a->ngram_max;
    p.cand_pos = a->cand_pos;
    p.C_cap = a->C_cap;
    p.cand_count = a->cand_count;
    p.match_len = a->match_len;
    p.H = a->H;
    p.d = a->d;
    p.h_seq_stride = a->h_seq_stride;
    p.threshold = a->threshold;
    p.h_scores = a->h_scores;
    p.best_h = a->best_h;
    p.best_h_score = a->best_h_score;
    p.A = a->A;
    p.a_bf16 = a->a_dtype == PLDP_BF16;
    p.R = a->R;
    p.a_row_stride = a->a_row_stride;
    p.a_seq_stride = a->a_seq_stride;
    p.row_idx = a->row_idx;
    p.n_sel = sel;
    p.agg = static_cast<int>(a->agg);
    p.a_scores = a->a_scores;
    p.best_a = a->best_a;
    p.best_a_score = a->best_a_score;
    p.draft_from = a->draft_from;
    p.K = a->K;
    p.draft = a->draft;
    p.draft_len = a->draft_len;
    p.status = a->status;
    p.rows_offset = (qbytes + 127) / 128 * 128;
    const size_t smem = p.rows_offset + static_cast<size_t>(sel) * sizeof(int64_t);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (!a->H) return launch_draft_step<NoHidden>(p, B, smem, s);
    if (a->h_dtype == PLDP_BF16) return launch_draft_step<__nv_bfloat16>(p, B, smem, s);
    return launch_draft_step<float>(p, B, smem, s);
}
