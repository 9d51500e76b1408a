// pldp_draft_step: the drafting half of a PLD+ step -- candidate search (Eq. 1
// with the longest-suffix n-gram rule), ranking by hidden states (Eq. 3) and/or
// by attentions (Eq. 2), and draft extraction (Sec. 4.3) -- in two short kernels.
//
// Both kernels are kept small on purpose.  Between decode steps the model's own
// traffic evicts this library's code from L2, so every distinct stretch of code a
// CTA reaches costs an instruction fetch from DRAM; a long multi-phase kernel with
// one CTA per SM pays that many times in series.  Short straight-line kernels
// with many CTAs pay it once, in parallel.
//
//  1. scan: a flat grid of (chunk, sequence) CTAs streams the contexts with
//     16-byte loads and appends every occurrence j of x_t, with its suffix-match
//     length m, to a short per-sequence list in the workspace ((j << 4) | m).
//     It also starts pulling into L2 what the rank kernel will read for each
//     occurrence (its hidden row, its attention values) and the query row.
//  2. rank: one CTA per sequence reads its list, takes n* = the largest m, orders
//     the occurrences with m >= n* by position (the candidate list), scores them
//     by hidden states on half its warps while the other half scores attentions,
//     and writes the draft.  It returns
//     the list's count to zero for the next call.  A list that overflowed (more
//     than kHitCap occurrences) is redone by an ordered rescan of the context
//     inside the CTA.
//
// The query row H_{t-1} depends only on seq_len: the rank kernel's bulk copy of
// it into shared memory is issued at entry and lands while the list is read.
// Results are those of pldp_find_candidates, pldp_rank_hidden,
// pldp_rank_attention and pldp_extract_draft called in turn (fp32 score sums may
// be split differently, so scores can differ in their last bits).
#include <type_traits>

#include "pldp_rank.cuh"
#include "pldp_scan.cuh"

namespace pldp {
namespace {

constexpr int kThreads = 256;
constexpr int kScanVec = 8;                                    // int4 loads per scan thread
constexpr int64_t kChunk = int64_t(kThreads) * kScanVec * 4;   // positions per scan CTA
constexpr int kHitCap = 256;                                   // occurrences kept per sequence
constexpr size_t kSeqWs = 16 + kHitCap * 4;                    // workspace bytes per sequence
constexpr size_t kMaxQueryBytes = 196608;
constexpr int kMaxSelRows = 8192;
constexpr int64_t kMaxPositions = int64_t(1) << 27;            // (j << 4) | m fits 31 bits

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
    bool h_bf16;
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
    int draft_from;       // 0: hidden choice, 1: attention choice
    int K;
    int32_t* draft;
    int32_t* draft_len;
    uint32_t* status;
    unsigned char* ws;    // kSeqWs per sequence: the count (u32), then kHitCap entries
    size_t rows_offset;   // byte offset of the attention row table in dynamic shared memory
};

__device__ __forceinline__ unsigned* hit_count(unsigned char* ws, int b) {
    return reinterpret_cast<unsigned*>(ws + static_cast<size_t>(b) * kSeqWs);
}
__device__ __forceinline__ int32_t* hit_list(unsigned char* ws, int b) {
    return reinterpret_cast<int32_t*>(ws + static_cast<size_t>(b) * kSeqWs + 16);
}

// ---- 1. scan -----------------------------------------------------------------------
__device__ __forceinline__ void prefetch_l2_bulk(const void* ptr, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(ptr), "r"(bytes) : "memory");
}
__device__ __forceinline__ void prefetch_l2(const void* ptr) {
    asm volatile("prefetch.global.L2 [%0];" ::"l"(ptr));
}

// The rank kernel reads, per occurrence j, the hidden row H_{j-1} and the
// attention values A[r, j]; the scan finds j several microseconds earlier, so the
// warp that found it starts pulling those lines into L2 (and their address
// translations into the TLBs) right away.  Warp-uniform call.
__device__ __forceinline__ void prefetch_candidate(const DraftParams& p, int b, int64_t j, int lane) {
    if (p.H && j >= 1 && lane == 0) {
        const size_t es = p.h_bf16 ? 2 : 4;
        const char* hrow = static_cast<const char*>(p.H) + (static_cast<int64_t>(b) * p.h_seq_stride + (j - 1) * p.d) * es;
        prefetch_l2_bulk(hrow, static_cast<uint32_t>(p.d * es));
    }
    if (p.A) {
        const size_t es = p.a_bf16 ? 2 : 4;
        const char* ab = static_cast<const char*>(p.A) + static_cast<int64_t>(b) * p.a_seq_stride * es;
        for (int k = lane; k < p.n_sel; k += 32) {
            const int r = p.row_idx ? __ldg(p.row_idx + k) : k;
            if (r >= 0 && r < p.R) prefetch_l2(ab + (static_cast<int64_t>(r) * p.a_row_stride + j) * es);
        }
    }
}

template <bool VEC>
__global__ void __launch_bounds__(kThreads) draft_scan_kernel(const DraftParams p) {
    pdl_enter();
    const int b = blockIdx.y;
    const int64_t L = p.seq_len[b];
    if (L < 2 || L > p.T_cap) return;                 // nothing to find; the rank kernel reports
    const int64_t t = L - 1;
    const int tid = threadIdx.x, lane = tid & 31;
    if (blockIdx.x == 0 && tid == 0 && p.H && t >= 2) {   // the query row H_{t-1}, for the rank kernel
        const size_t es = p.h_bf16 ? 2 : 4;
        prefetch_l2_bulk(static_cast<const char*>(p.H) + (static_cast<int64_t>(b) * p.h_seq_stride + (t - 1) * p.d) * es,
                         static_cast<uint32_t>(p.d * es));
    }
    const int64_t c0 = static_cast<int64_t>(blockIdx.x) * kChunk;
    const int64_t c1 = c0 + kChunk < t ? c0 + kChunk : t;
    if (c0 >= c1) return;
    const int32_t* row = p.ids + static_cast<int64_t>(b) * p.ids_stride;
    const int32_t xt = __ldg(row + t);

    // Each thread covers 4 * kScanVec positions; bit i of `mask` marks its i-th.
    uint32_t mask = 0;
    if constexpr (VEC) {
        const int4* row4 = reinterpret_cast<const int4*>(row);
        const int64_t q0 = c0 >> 2, q1 = (c1 + 3) >> 2;
        int4 v[kScanVec];
#pragma unroll
        for (int u = 0; u < kScanVec; ++u) {
            const int64_t q = q0 + tid + u * kThreads;
            if (q < q1) v[u] = __ldg(row4 + q);
        }
#pragma unroll
        for (int u = 0; u < kScanVec; ++u) {
            const int64_t q = q0 + tid + u * kThreads;
            if (q >= q1) continue;
            const int32_t e[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (e[k] == xt && 4 * q + k < c1) mask |= 1u << (4 * u + k);
        }
    } else {
        int32_t v[kScanVec * 4];
#pragma unroll
        for (int u = 0; u < kScanVec * 4; ++u) {
            const int64_t j = c0 + tid + u * kThreads;
            if (j < c1) v[u] = __ldg(row + j);
        }
#pragma unroll
        for (int u = 0; u < kScanVec * 4; ++u) {
            const int64_t j = c0 + tid + u * kThreads;
            if (j < c1 && v[u] == xt) mask |= 1u << u;
        }
    }
    // Occurrences, one at a time per warp: prefetch for the rank kernel, then record.
    unsigned pending = __ballot_sync(0xFFFFFFFFu, mask != 0);
    while (pending) {
        const int src = __ffs(pending) - 1;
        const uint32_t m_src = __shfl_sync(0xFFFFFFFFu, mask, src);
        const int bit = __ffs(m_src) - 1;
        int64_t j;
        if constexpr (VEC) {
            const int64_t q = (c0 >> 2) + (tid - lane + src) + (bit >> 2) * kThreads;
            j = 4 * q + (bit & 3);
        } else {
            j = c0 + (tid - lane + src) + static_cast<int64_t>(bit) * kThreads;
        }
        unsigned slot = 0;
        if (lane == src) {
            const int m = suffix_match(row, j, t, p.ngram_max);
            slot = atomicAdd(hit_count(p.ws, b), 1u);
            if (slot < kHitCap) hit_list(p.ws, b)[slot] = static_cast<int32_t>((j << 4) | m);
            mask &= mask - 1;
        }
        // Past kHitCap the rank kernel rescans; prefetching stops there too.
        if (__shfl_sync(0xFFFFFFFFu, slot, src) < kHitCap) prefetch_candidate(p, b, j, lane);
        pending = __ballot_sync(0xFFFFFFFFu, mask != 0);
    }
}

// ---- 2. rank -----------------------------------------------------------------------
struct ListState {
    int32_t sorted[kHitCap];   // the candidate list, in order
    int32_t raw[kHitCap];      // the recorded occurrences, (j << 4) | m
    int nstar, total;
};

template <typename TH, bool IVEC>
__global__ void __launch_bounds__(kThreads) draft_rank_kernel(const DraftParams p) {
    constexpr bool HAS_H = !std::is_same<TH, NoHidden>::value;
    using TQ = typename std::conditional<HAS_H, TH, float>::type;
    extern __shared__ __align__(128) unsigned char dyn_smem[];
    TQ* q_sh = reinterpret_cast<TQ*>(dyn_smem);                                   // H_{t-1}
    int64_t* rows_sh = reinterpret_cast<int64_t*>(dyn_smem + p.rows_offset);     // attention rows
    __shared__ ListState ls;
    __shared__ ScanShared ss;
    __shared__ RankShared hs, as;
    __shared__ __align__(8) uint64_t q_bar;
    __shared__ int bad_rows;

    pdl_enter();
    const int b = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const bool has_a = p.A != nullptr;
    const int64_t L = p.seq_len[b];
    const bool valid = L >= 0 && L <= p.T_cap;
    const int64_t t = L - 1;
    const int32_t* row = p.ids + static_cast<int64_t>(b) * p.ids_stride;
    const bool q_fetch = HAS_H && valid && t >= 2;
    const TQ* hb = nullptr;
    if constexpr (HAS_H) {
        hb = static_cast<const TQ*>(p.H) + static_cast<int64_t>(b) * p.h_seq_stride;
        if (q_fetch && tid == 0) {
            const uint32_t qbytes = static_cast<uint32_t>(p.d * sizeof(TQ));
            mbar_init(&q_bar, 1);
            fence_mbar_init();
            mbar_arrive_expect_tx(&q_bar, qbytes);
            bulk_g2s(q_sh, hb + (t - 1) * p.d, qbytes, &q_bar);
        }
    }
    unsigned* cnt_g = hit_count(p.ws, b);
    const unsigned nh = __ldcg(cnt_g);
    rank_shared_init(hs);
    rank_shared_init(as);
    if (tid <= PLDP_MAX_NGRAM) ss.cnt[tid] = 0;
    const bool listed = nh <= static_cast<unsigned>(kHitCap);
    if (valid && listed)
        for (int i = tid; i < static_cast<int>(nh); i += kThreads) ls.raw[i] = __ldcg(hit_list(p.ws, b) + i);
    bool bad = false;
    if (has_a && valid) bad = stage_rows(rows_sh, p.row_idx, p.n_sel, p.R, p.a_row_stride, &bad_rows);
    __syncthreads();
    if (tid == 0) *cnt_g = 0u;                        // ready for the next call

    if (!valid) {
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
        return;
    }

    // ---- the candidate list ------------------------------------------------------------
    int32_t* cand_row = p.cand_pos + static_cast<int64_t>(b) * p.C_cap;
    if (listed) {
        if (tid == 0) {
            int mx = 0;
            for (int i = 0; i < static_cast<int>(nh); ++i) mx = max(mx, ls.raw[i] & 15);
            const int nstar = mx >= p.ngram_min ? mx : 0;
            int total = 0;
            if (nstar)
                for (int i = 0; i < static_cast<int>(nh); ++i) total += ((ls.raw[i] & 15) >= nstar) ? 1 : 0;
            ls.nstar = nstar;
            ls.total = total;
        }
        __syncthreads();
        const int nstar = ls.nstar;
        if (nstar > 0)
            for (int i = tid; i < static_cast<int>(nh); i += kThreads) {
                const int32_t e = ls.raw[i];
                if ((e & 15) < nstar) continue;
                int r = 0;                              // positions are distinct: so are ranks
                for (int k = 0; k < static_cast<int>(nh); ++k) {
                    const int32_t f = ls.raw[k];
                    r += ((f & 15) >= nstar && f < e) ? 1 : 0;
                }
                ls.sorted[r] = e >> 4;
            }
        __syncthreads();
    } else {
        // more occurrences than the list holds: an ordered rescan of the whole context
        int c[PLDP_MAX_NGRAM];
#pragma unroll
        for (int k = 0; k < PLDP_MAX_NGRAM; ++k) c[k] = 0;
        scan_count<IVEC>(GlobalIds{row}, row, 0, t, t, p.ngram_max, c);
        scan_reduce_counts(c, p.ngram_max, ss);
        __syncthreads();
        if (tid == 0) {
            int nstar = 0, total = 0;
            for (int n = p.ngram_max; n >= p.ngram_min; --n)
                if (ss.cnt[n] > 0) {
                    nstar = n;
                    total = ss.cnt[n];
                    break;
                }
            ss.nstar = nstar;
            ss.total = total;
            ss.offset = 0;
            ss.mine = total;
            ls.nstar = nstar;
            ls.total = total;
        }
        __syncthreads();
        scan_write<IVEC>(GlobalIds{row}, row, 0, t, t, p.ngram_max, ss, cand_row, p.C_cap);
    }
    const int total = ls.total;
    const int n = total < p.C_cap ? total : p.C_cap;
    if (listed)
        for (int i = tid; i < n; i += kThreads) cand_row[i] = ls.sorted[i];
    if (tid == 0) {
        p.cand_count[b] = total;
        p.match_len[b] = ls.nstar;
        if (p.status && total > p.C_cap) atomicOr(p.status + b, PLDP_ST_CAND_OVERFLOW);
        if (bad && p.status) atomicOr(p.status + b, PLDP_ST_ROW_INDEX);
    }
    __syncthreads();                                   // cand_row is complete for the rescan path

    // ---- ranking: hidden states on warps 0-3 while attentions run on warps 4-7 ----------
    const bool split = HAS_H && has_a;
    const WarpGroup hg = split ? WarpGroup{0, 4, 1} : whole_cta();
    const WarpGroup ag = split ? WarpGroup{4, 4, 2} : whole_cta();
    if constexpr (HAS_H) {
        if (!split || warp < 4) {
            float* hsc = p.h_scores ? p.h_scores + static_cast<int64_t>(b) * p.C_cap : nullptr;
            if (listed)
                hidden_rank_cta<TQ, true, true>(hb, p.d, t, ls.sorted, n, 1, 0, nullptr, q_sh, &q_bar, q_fetch,
                                                p.threshold, hsc, hs, hg);
            else
                hidden_rank_cta<TQ, true, false>(hb, p.d, t, cand_row, n, 1, 0, nullptr, q_sh, &q_bar,
                                                 q_fetch, p.threshold, hsc, hs, hg);
            if (q_fetch && tid == 0 && !mbar_wait(&q_bar, 0, kMbarPolls)) hs.err = 1;   // landed before exit
        }
    }
    if (has_a && (!split || warp >= 4)) {
        const size_t es = p.a_bf16 ? 2 : 4;
        const void* ab = static_cast<const char*>(p.A) + static_cast<int64_t>(b) * p.a_seq_stride * es;
        float* asc = p.a_scores ? p.a_scores + static_cast<int64_t>(b) * p.C_cap : nullptr;
        if (listed)
            attention_rank_cta<true>(ab, p.a_bf16, rows_sh, p.n_sel, t, ls.sorted, n, 1, 0, nullptr,
                                     p.agg == PLDP_AGG_MAX, asc, as, ag);
        else
            attention_rank_cta<false>(ab, p.a_bf16, rows_sh, p.n_sel, t, cand_row, n, 1, 0, nullptr,
                                      p.agg == PLDP_AGG_MAX, asc, as, ag);
    }
    __syncthreads();

    // ---- best and draft (warp 0) -----------------------------------------------------------
    if (warp == 0) {
        const unsigned long long hk = rank_best_key(hs), ak = rank_best_key(as);
        const int err = hs.err;
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
        for (int i = lane; i < p.K; i += 32)
            p.draft[static_cast<int64_t>(b) * p.K + i] = (i < dl) ? __ldg(row + js + 1 + i) : -1;
        if (tid == 0) p.draft_len[b] = static_cast<int32_t>(dl);
    }
}

template <typename TH, bool IVEC>
pldp_status launch_t(const DraftParams& p, int B, size_t smem, cudaStream_t s) {
    const int64_t chunks = (p.T_cap + kChunk - 1) / kChunk;
    if (chunks > 65535) return fail(PLDP_ERR_UNSUPPORTED, "draft_step: T_cap too large for the scan grid");
    if (chunks > 0) {
        cudaError_t e = launch_pdl(draft_scan_kernel<IVEC>, dim3(static_cast<unsigned>(chunks), static_cast<unsigned>(B)),
                                   dim3(kThreads), 0, s, 0, p);
        if (e != cudaSuccess)
            return fail(PLDP_ERR_CUDA, "draft_step (scan): launch failed: %s", cudaGetErrorString(e));
    }
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(draft_rank_kernel<TH, IVEC>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess)
            return fail(PLDP_ERR_CUDA, "draft_step: shared memory attribute: %s", cudaGetErrorString(e));
    }
    cudaError_t e = launch_pdl(draft_rank_kernel<TH, IVEC>, dim3(static_cast<unsigned>(B)), dim3(kThreads), smem, s,
                               0, p);
    if (e != cudaSuccess)
        return fail(PLDP_ERR_CUDA, "draft_step (rank): launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}

template <typename TH>
pldp_status launch_draft_step(const DraftParams& p, int B, size_t smem, cudaStream_t s, bool ivec) {
    return ivec ? launch_t<TH, true>(p, B, smem, s) : launch_t<TH, false>(p, B, smem, s);
}

}  // namespace
}  // namespace pldp

using namespace pldp;

extern "C" PLDP_API size_t pldp_draft_workspace_size(int B) {
    return B < 0 ? 0 : static_cast<size_t>(B) * kSeqWs;
}

extern "C" PLDP_API pldp_status pldp_draft_step(const pldp_draft_step_args* a, void* stream) {
    if (!a) return fail(PLDP_ERR_INVALID_ARG, "draft_step: null argument block");
    const int B = a->B;
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "draft_step: B < 0");
    if (B > 65535) return fail(PLDP_ERR_UNSUPPORTED, "draft_step: B > 65535");
    if (a->T_cap < 0 || a->T_cap > kMaxPositions)
        return fail(PLDP_ERR_INVALID_ARG, "draft_step: T_cap outside [0, 2^27]");
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
    if (!a->workspace || a->workspace_bytes < pldp_draft_workspace_size(B) || !aligned16(a->workspace))
        return fail(PLDP_ERR_INVALID_ARG, "draft_step: workspace needs %zu bytes, 16-byte aligned",
                    pldp_draft_workspace_size(B));
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
    p.h_bf16 = a->h_dtype == PLDP_BF16;
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
    p.ws = static_cast<unsigned char*>(a->workspace);
    p.rows_offset = (qbytes + 127) / 128 * 128;
    const size_t smem = p.rows_offset + static_cast<size_t>(sel) * sizeof(int64_t);
    const bool ivec = aligned16(a->ids) && a->ids_stride % 4 == 0 && a->T_cap % 4 == 0;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (!a->H) return launch_draft_step<NoHidden>(p, B, smem, s, ivec);
    if (a->h_dtype == PLDP_BF16) return launch_draft_step<__nv_bfloat16>(p, B, smem, s, ivec);
    return launch_draft_step<float>(p, B, smem, s, ivec);
}
