// pldp_draft_step: the drafting half of a PLD+ step -- candidate search (Eq. 1
// with the longest-suffix n-gram rule), ranking by hidden states (Eq. 3) and/or
// by attentions (Eq. 2), and draft extraction (Sec. 4.3) -- in one launch; and
// pldp_verify_greedy_draft / pldp_verify_sample_draft: greedy or sampling
// verification (Sec. 4.4) followed by the next step's drafting.  Three kernels:
//  * draft_step_kernel scans the contexts (below);
//  * draft_index_kernel looks the occurrences up in the incremental token index
//    (further down), one CTA per sequence;
//  * verify_draft_kernel runs the finish of verification (on the greedy pass's
//    row keys, or on the draws of sampling) and then the indexed drafting in the
//    same CTA.
//
// The scanning kernel: a flat grid of (chunk, sequence) CTAs.  Each CTA
//  1. streams its chunk of the context with 16-byte loads and, for every
//     occurrence j of x_t, takes the suffix-match length m and a slot in a short
//     per-sequence list held in the workspace;
//  2. scores each occurrence it found with all its threads -- cos(H_{j-1},
//     H_{t-1}) and the max (or sum) of the selected attention rows at key j, both
//     in one round trip to memory -- and stores (j, m, scores) in the slot;
//  3. takes a ticket.  The CTA that takes a sequence's last ticket finishes it:
//     it reads the list, takes n* = the largest m, orders the occurrences with
//     m >= n* by position (the candidate list), picks the best of each ranking
//     from the stored scores, writes the draft, and returns the list's header to
//     zero for the next call.
// No CTA waits for another.  Occurrences are scored before n* is known, so
// those with m < n* are scored for nothing; they are few.  A list that
// overflowed (more than kHitCap occurrences) is redone by the finishing CTA: an
// ordered rescan of the context, then the same scorer per candidate.
//
// Every score comes from the same CTA-wide reduction (a fixed share per thread,
// partial sums combined in warp order), whichever CTA computes it, so results
// are deterministic.  Results are those of pldp_find_candidates,
// pldp_rank_hidden, pldp_rank_attention and pldp_extract_draft called in turn
// (fp32 score sums are split differently, so scores can differ in their last
// bits).
#include <climits>
#include <type_traits>

#include "pldp_rank.cuh"
#include "pldp_scan.cuh"
#include "pldp_verify.cuh"

namespace pldp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kScanVec = 9;                                    // int4 loads per scan thread
constexpr int64_t kChunk = int64_t(kThreads) * kScanVec * 4;   // positions per CTA
constexpr int kHitCap = 256;                                   // occurrences kept per sequence
constexpr size_t kSeqWs = 16 + kHitCap * 16;                   // header + 16-byte entries
constexpr int kScoreUnroll = 2;                                // 16-byte row loads in flight
constexpr int kScoreBatch = 2;                                 // occurrences scored per pass (scan kernel)
constexpr int kMaxScoreBatch = 4;                              // ... and at most (the indexed kernel)
constexpr int kSpeculate = kMaxScoreBatch;                     // occurrences scored before their suffix match
constexpr int kPrefetchOcc = 32;                                // occurrences whose rows are prefetched otherwise
constexpr size_t kMaxQueryBytes = 196608;
constexpr int kMaxSelRows = 8192;
constexpr int64_t kMaxPositions = int64_t(1) << 27;            // (j << 4) | m fits 31 bits

static_assert(kHitCap <= kThreads, "the finish gives each list entry its own thread");

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
    int64_t a_key_stride;
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
    unsigned char* ws;    // kSeqWs per sequence: count, ticket (u32 each), pad; entries
};

// Workspace of sequence b: header[0] = occurrences recorded, header[1] = tickets
// taken; entry i = ((j << 4) | m, hidden score bits, attention score bits, 0).
__device__ __forceinline__ unsigned* seq_header(unsigned char* ws, int b) {
    return reinterpret_cast<unsigned*>(ws + static_cast<size_t>(b) * kSeqWs);
}
__device__ __forceinline__ uint4* seq_entries(unsigned char* ws, int b) {
    return reinterpret_cast<uint4*>(ws + static_cast<size_t>(b) * kSeqWs + 16);
}

struct Hit {
    int32_t j, m;
};

// Warp reduce-scatter of N values (N a power of two, <= 32): at each butterfly
// level a lane keeps half of its values and trades the other half with its
// partner, so the N totals take N - 1 + 5 - log2(N) shuffles instead of 5 N.
// Returns the total (sum, or max when use_max) of value lane >> (5 - log2 N).
// Every total is formed in one fixed order, the same in every lane holding it.
template <int N>
__device__ __forceinline__ float warp_reduce_scatter(float (&v)[N], bool use_max) {
    static_assert(N >= 1 && N <= 32 && (N & (N - 1)) == 0, "N: a power of two up to 32");
    constexpr int LOG2N = N >= 32 ? 5 : N >= 16 ? 4 : N >= 8 ? 3 : N >= 4 ? 2 : N >= 2 ? 1 : 0;
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int s = 0; s < LOG2N; ++s) {
        const int n = N >> s, o = 16 >> s;
        const bool upper = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < N / 2; ++i) {
            if (i >= n / 2) continue;
            const float keep = upper ? v[i + n / 2] : v[i];
            const float send = upper ? v[i] : v[i + n / 2];
            const float got = __shfl_xor_sync(0xFFFFFFFFu, send, o);
            v[i] = use_max ? fmaxf(keep, got) : keep + got;
        }
    }
    float r = v[0];
#pragma unroll
    for (int o = 16 >> LOG2N; o > 0; o >>= 1) {
        const float got = __shfl_xor_sync(0xFFFFFFFFu, r, o);
        r = use_max ? fmaxf(r, got) : r + got;
    }
    return r;
}

template <int NB>
__device__ __forceinline__ float (&part_buf(float (&part)[kMaxScoreBatch][kWarps][4]))[NB][kWarps][4] {
    return *reinterpret_cast<float(*)[NB][kWarps][4]>(&part[0]);
}

struct StepShared {
    Hit hit[kHitCap];                        // occurrences this CTA found (the first kHitCap)
    alignas(16) float part[2][kMaxScoreBatch][kWarps][4];   // per-warp partials: dot, |a|^2, |q|^2, attention
    int32_t jl[kHitCap];                     // finish: positions of the candidates (else INT_MAX)
    unsigned long long wkey[2][kWarps];      // finish: per-warp best keys (hidden, attention)
    int wmax[kWarps];
    int32_t suf[PLDP_MAX_NGRAM];             // x_t, x_{t-1}, ... (n_max of them)
    int nhit, skip, last;
    ScanShared ss;                           // finish: the ordered rescan of an overflowed list
};

// Eq. 3 and Eq. 2 for candidates j[0 .. nb) of sequence b (nb <= NB), by all
// threads of the CTA: thread i takes 16-byte chunks i, i + 256, ... of H_{j-1}
// and H_{t-1} and selected rows i, i + 256, ...; partial sums meet in `part`
// and are combined in warp order.  The candidates of one pass share the loads of
// H_{t-1} and are otherwise independent: a score does not depend on which pass
// or slot computes it.  The attention values of each thread's first selected row
// are loaded before the hidden rows are used, so both arrive in one round trip.
// Scores are returned in thread 0: the cosine (-inf when j = 0 has no H_{j-1})
// and the attention max / sum.  CTA-uniform call with one barrier; callers
// alternate `part` buffers.
template <typename TH, int NB>
__device__ __forceinline__ void cta_score(const DraftParams& p, int b, const int64_t (&j)[NB], int nb, int64_t t,
                                          float (&part)[NB][kWarps][4], float (&s_h)[NB], float (&s_a)[NB]) {
    constexpr bool HAS_H = !std::is_same<TH, NoHidden>::value;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const bool is_max = p.agg == PLDP_AGG_MAX;
    bool h_ok[NB], a_ok[NB];
    bool any_h = false;
#pragma unroll
    for (int h = 0; h < NB; ++h) {
        h_ok[h] = HAS_H && h < nb && j[h] >= 1 && j[h] < t;
        a_ok[h] = p.A != nullptr && h < nb && j[h] >= 0 && j[h] < t;
        any_h |= h_ok[h];
    }
    float dot[NB], na[NB], nq = 0.f, acc[NB];
#pragma unroll
    for (int h = 0; h < NB; ++h) {
        dot[h] = 0.f;
        na[h] = 0.f;
        acc[h] = is_max ? -INFINITY : 0.0f;
    }
    const size_t a_es = p.a_bf16 ? 2 : 4;
    const void* ab = p.A ? static_cast<const char*>(p.A) + static_cast<int64_t>(b) * p.a_seq_stride * a_es : nullptr;
    float av[NB];                                                 // selected row `tid`, in flight with H
    {
        const int r = (p.A != nullptr && tid < p.n_sel) ? (p.row_idx ? __ldg(p.row_idx + tid) : tid) : -1;
        const bool rv = r >= 0 && r < p.R;
#pragma unroll
        for (int h = 0; h < NB; ++h)
            av[h] = (rv && a_ok[h]) ? load_attn(ab, static_cast<int64_t>(r) * p.a_row_stride + j[h] * p.a_key_stride, p.a_bf16) : NAN;
    }
    if constexpr (HAS_H) {
        if (any_h) {
            constexpr int E = 16 / sizeof(TH);
            const TH* hb = static_cast<const TH*>(p.H) + static_cast<int64_t>(b) * p.h_seq_stride;
            const TH* qrow = hb + (t - 1) * p.d;                  // H_{t-1}
            const TH* arow[NB];
#pragma unroll
            for (int h = 0; h < NB; ++h) arow[h] = h_ok[h] ? hb + (j[h] - 1) * p.d : qrow;   // H_{j-1}
            const int64_t nch = p.d / E;
            for (int64_t c0 = tid; c0 < nch; c0 += static_cast<int64_t>(kThreads) * kScoreUnroll) {
                uint4 q[kScoreUnroll], a[NB][kScoreUnroll];
#pragma unroll
                for (int u = 0; u < kScoreUnroll; ++u) {
                    const int64_t c = c0 + static_cast<int64_t>(kThreads) * u;
                    if (c < nch) {
                        q[u] = ld_stream16(qrow + c * E);
#pragma unroll
                        for (int h = 0; h < NB; ++h)
                            if (h_ok[h]) a[h][u] = ld_stream16(arow[h] + c * E);
                    }
                }
#pragma unroll
                for (int u = 0; u < kScoreUnroll; ++u) {
                    if (c0 + static_cast<int64_t>(kThreads) * u >= nch) continue;
                    float dead0 = 0.f, dead1 = 0.f;                 // |H_{t-1}|^2 once for the pass
                    accum16<TH>(q[u], q[u], dead0, dead1, nq);
#pragma unroll
                    for (int h = 0; h < NB; ++h) {
                        float dead2 = 0.f;
                        if (h_ok[h]) accum16<TH>(a[h][u], q[u], dot[h], na[h], dead2);
                    }
                }
            }
        }
    }
    if (p.A != nullptr) {
#pragma unroll
        for (int h = 0; h < NB; ++h)
            if (av[h] == av[h]) acc[h] = is_max ? fmaxf(acc[h], av[h]) : acc[h] + av[h];
        for (int k = tid + kThreads; k < p.n_sel; k += kThreads) {
            const int r = p.row_idx ? __ldg(p.row_idx + k) : k;
            const bool rv = r >= 0 && r < p.R;
            float v[NB];
#pragma unroll
            for (int h = 0; h < NB; ++h)
                v[h] = (rv && a_ok[h]) ? load_attn(ab, static_cast<int64_t>(r) * p.a_row_stride + j[h] * p.a_key_stride, p.a_bf16) : NAN;
#pragma unroll
            for (int h = 0; h < NB; ++h)
                if (v[h] == v[h]) acc[h] = is_max ? fmaxf(acc[h], v[h]) : acc[h] + v[h];
        }
    }
    // warp totals by reduce-scatter: lane l ends with one of them
    if constexpr (HAS_H) {
        float w[2 * NB];                                          // dot products, then |H_{j-1}|^2
#pragma unroll
        for (int h = 0; h < NB; ++h) {
            w[h] = dot[h];
            w[NB + h] = na[h];
        }
        const float tw = warp_reduce_scatter<2 * NB>(w, false);
        constexpr int SW = 32 / (2 * NB);                         // lanes holding each total
        const int iw = lane / SW;
        if (lane % SW == 0) part[iw % NB][warp][iw < NB ? 0 : 1] = tw;
        nq = warp_sum(nq);
        if (lane < NB) part[lane][warp][2] = nq;
    } else {
        if (lane < NB) part[lane][warp][0] = part[lane][warp][1] = part[lane][warp][2] = 0.f;
    }
    {
        const float ta = warp_reduce_scatter<NB>(acc, is_max);
        constexpr int SA = 32 / NB;
        if (lane % SA == 0) part[lane / SA][warp][3] = ta;
    }
    __syncthreads();
    if (warp == 0) {
        // lane (h, w) = (lane / kWarps, lane % kWarps) takes warp w's partials of
        // candidate h; the kWarps lanes of a candidate combine them in a fixed tree
        static_assert(NB * kWarps <= 32, "a lane per (candidate, warp)");
        const int h = lane / kWarps, w = lane % kWarps;
        float4 v = make_float4(0.f, 0.f, 0.f, is_max ? -INFINITY : 0.f);
        if (h < NB) v = *reinterpret_cast<const float4*>(&part[h][w][0]);
#pragma unroll
        for (int o = kWarps / 2; o > 0; o >>= 1) {
            v.x += __shfl_xor_sync(0xFFFFFFFFu, v.x, o);
            v.y += __shfl_xor_sync(0xFFFFFFFFu, v.y, o);
            v.z += __shfl_xor_sync(0xFFFFFFFFu, v.z, o);
            const float x = __shfl_xor_sync(0xFFFFFFFFu, v.w, o);
            v.w = is_max ? fmaxf(v.w, x) : v.w + x;
        }
        bool hv = false, avl = false;
#pragma unroll
        for (int k = 0; k < NB; ++k)
            if (k == h) {
                hv = h_ok[k];
                avl = a_ok[k];
            }
        const float sh_ = hv ? finish_cosine(v.x, v.y, v.z) : -INFINITY;
        const float sa_ = avl ? v.w : -INFINITY;
#pragma unroll
        for (int k = 0; k < NB; ++k) {
            s_h[k] = __shfl_sync(0xFFFFFFFFu, sh_, k * kWarps);
            s_a[k] = __shfl_sync(0xFFFFFFFFu, sa_, k * kWarps);
        }
    }
}

// The finish of a sequence whose occurrences were not gathered (an overflowed
// list, or a token the index cannot answer for): an ordered rescan of the
// context writes the candidate list, the candidates' hidden rows start towards
// L2, then the candidates are scored by cta_score, NB per pass.  Kept out of
// line: its registers do not weigh on the common path.  CTA-uniform call; keys
// are left in thread 0.
template <typename TH, bool IVEC, int NB, typename RD = ReadOnlyIds>
__device__ __noinline__ void finish_overflow(const DraftParams& p, int b, int64_t t, const int32_t* row,
                                             int32_t* cand_row, float* hsc, float* asc, StepShared& sh,
                                             unsigned long long& hk, unsigned long long& ak, int& nstar,
                                             int& total) {
    constexpr bool HAS_H = !std::is_same<TH, NoHidden>::value;
    const bool has_a = p.A != nullptr;
    const int tid = threadIdx.x;
    int c[PLDP_MAX_NGRAM];
#pragma unroll
    for (int k = 0; k < PLDP_MAX_NGRAM; ++k) c[k] = 0;
    scan_count<IVEC, GlobalIdsT<RD>, RD>(GlobalIdsT<RD>{row}, row, 0, t, t, p.ngram_max, c);
    scan_reduce_counts(c, p.ngram_max, sh.ss);
    __syncthreads();
    if (tid == 0) {
        int ns = 0, tot = 0;
        for (int n = p.ngram_max; n >= p.ngram_min; --n)
            if (sh.ss.cnt[n] > 0) {
                ns = n;
                tot = sh.ss.cnt[n];
                break;
            }
        sh.ss.nstar = ns;
        sh.ss.total = tot;
        sh.ss.offset = 0;
        sh.ss.mine = tot;
    }
    __syncthreads();
    nstar = sh.ss.nstar;
    total = sh.ss.total;
    scan_write<IVEC, GlobalIdsT<RD>, NoHook, RD>(GlobalIdsT<RD>{row}, row, 0, t, t, p.ngram_max, sh.ss, cand_row,
                                                 p.C_cap);
    __syncthreads();
    const int n = total < p.C_cap ? total : p.C_cap;
    if (HAS_H && n > NB) {
        const size_t h_es = p.h_bf16 ? 2 : 4;
        for (int i = tid; i < n; i += kThreads) {
            const int64_t j = __ldcg(cand_row + i);
            if (j >= 1 && j < t)
                prefetch_l2_bulk(static_cast<const char*>(p.H) + (static_cast<int64_t>(b) * p.h_seq_stride + (j - 1) * p.d) * h_es,
                                 static_cast<uint32_t>(p.d * h_es));
        }
    }
    for (int i0 = 0; i0 < n; i0 += NB) {
        const int nb = n - i0 < NB ? n - i0 : NB;
        int64_t j[NB];
#pragma unroll
        for (int h = 0; h < NB; ++h) j[h] = h < nb ? __ldcg(cand_row + i0 + h) : -1;
        float s_h[NB], s_a[NB];
        cta_score<TH, NB>(p, b, j, nb, t, part_buf<NB>(sh.part[(i0 / NB) & 1]), s_h, s_a);
        if (tid == 0)
            for (int h = 0; h < nb; ++h) {
                const int i = i0 + h;
                if (HAS_H) {
                    if (hsc) hsc[i] = s_h[h];
                    if (j[h] >= 1 && s_h[h] > p.threshold) {
                        const unsigned long long key = pack_key(s_h[h], static_cast<uint32_t>(j[h]));
                        hk = key > hk ? key : hk;
                    }
                }
                if (has_a) {
                    if (asc) asc[i] = s_a[h];
                    const unsigned long long key = pack_key(s_a[h], static_cast<uint32_t>(j[h]));
                    ak = key > ak ? key : ak;
                }
            }
    }
}

template <typename TH, bool IVEC>
__global__ void __launch_bounds__(kThreads, 4) draft_step_kernel(const DraftParams p) {
    constexpr bool HAS_H = !std::is_same<TH, NoHidden>::value;
    __shared__ StepShared sh;
    pdl_enter();
    const int b = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t L = p.seq_len[b];
    const bool valid = L >= 0 && L <= p.T_cap;
    const int64_t t = L - 1;
    const int32_t* row = p.ids + static_cast<int64_t>(b) * p.ids_stride;
    unsigned* hdr = seq_header(p.ws, b);
    const size_t h_es = p.h_bf16 ? 2 : 4;
    // The chunk's ids do not depend on seq_len: their loads go out first, bounded
    // by the row's capacity, and land while seq_len and the suffix arrive.
    const int64_t c0 = static_cast<int64_t>(blockIdx.x) * kChunk;
    const int64_t ce = c0 + kChunk < p.T_cap ? c0 + kChunk : p.T_cap;
    constexpr int NV = IVEC ? kScanVec : kScanVec * 4;
    using VT = typename std::conditional<IVEC, int4, int32_t>::type;
    VT v[NV];
#pragma unroll
    for (int u = 0; u < NV; ++u) {
        if constexpr (IVEC) {
            const int64_t q = (c0 >> 2) + tid + u * kThreads;
            if (q < (ce >> 2)) v[u] = __ldg(reinterpret_cast<const int4*>(row) + q);
        } else {
            const int64_t j = c0 + tid + u * kThreads;
            if (j < ce) v[u] = __ldg(row + j);
        }
    }
    if (tid < PLDP_MAX_NGRAM)                                     // x_t and the n_max - 1 tokens before it
        sh.suf[tid] = (valid && tid < p.ngram_max && t - tid >= 0) ? __ldg(row + t - tid) : 0;
    if (tid == 0) {
        sh.nhit = 0;
        if (HAS_H && valid && t >= 2 && blockIdx.x == 0)        // H_{t-1}: every scored candidate reads it
            prefetch_l2_bulk(static_cast<const char*>(p.H) + (static_cast<int64_t>(b) * p.h_seq_stride + (t - 1) * p.d) * h_es,
                             static_cast<uint32_t>(p.d * h_es));
    }
    __syncthreads();

    // ---- 1. scan this chunk for x_t ------------------------------------------------------
    const int64_t c1 = c0 + kChunk < t ? c0 + kChunk : t;
    if (valid && t >= 1 && c0 < c1) {
        const int32_t xt = sh.suf[0];
        uint64_t mask = 0;                                        // bit i: this thread's i-th position
#pragma unroll
        for (int u = 0; u < NV; ++u) {
            if constexpr (IVEC) {
                const int64_t q = (c0 >> 2) + tid + u * kThreads;
                const int32_t e[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    if (e[k] == xt && 4 * q + k < c1) mask |= 1ull << (4 * u + k);
            } else {
                const int64_t j = c0 + tid + u * kThreads;
                if (j < c1 && v[u] == xt) mask |= 1ull << u;
            }
        }
        while (mask) {                                            // rarely more than one
            const int bit = __ffsll(static_cast<long long>(mask)) - 1;
            mask &= mask - 1;
            int64_t j;
            if constexpr (IVEC)
                j = 4 * ((c0 >> 2) + tid + (bit >> 2) * kThreads) + (bit & 3);
            else
                j = c0 + tid + static_cast<int64_t>(bit) * kThreads;
            int m = 1;                                            // common suffix of x[..j] and x[..t]
            while (m < p.ngram_max && j - m >= 0 && __ldg(row + j - m) == sh.suf[m]) ++m;
            const int k = atomicAdd(&sh.nhit, 1);
            if (k < kHitCap) {                                    // more: the list overflows anyway
                sh.hit[k] = Hit{static_cast<int32_t>(j), m};
                if (HAS_H && j >= 1)
                    prefetch_l2_bulk(static_cast<const char*>(p.H) +
                                         (static_cast<int64_t>(b) * p.h_seq_stride + (j - 1) * p.d) * h_es,
                                     static_cast<uint32_t>(p.d * h_es));
            }
        }
    }
    __syncthreads();

    // ---- 2. score what this CTA found ----------------------------------------------------
    // One atomic reserves the CTA's slots in the sequence's list; its answer is
    // needed only when the entries are written, so it runs under the scoring.
    const int nhit = sh.nhit;
    if (nhit > 0) {
        unsigned base = 0;
        if (tid == 0) base = atomicAdd(hdr, static_cast<unsigned>(nhit));
        if (nhit > 8) {                                           // skip the scores of a list that overflowed
            if (tid == 0) sh.skip = base + static_cast<unsigned>(nhit) > static_cast<unsigned>(kHitCap);
            __syncthreads();
        }
        if (nhit <= 8 || !sh.skip)                                // (nhit > kHitCap always skips)
            for (int k = 0; k < nhit; k += kScoreBatch) {
                const int nb = nhit - k < kScoreBatch ? nhit - k : kScoreBatch;
                int64_t j[kScoreBatch];
#pragma unroll
                for (int h = 0; h < kScoreBatch; ++h) j[h] = h < nb ? sh.hit[k + h].j : -1;
                float s_h[kScoreBatch], s_a[kScoreBatch];
                cta_score<TH, kScoreBatch>(p, b, j, nb, t, part_buf<kScoreBatch>(sh.part[(k / kScoreBatch) & 1]), s_h,
                                           s_a);
                if (tid == 0)
                    for (int h = 0; h < nb; ++h) {
                        const Hit e = sh.hit[k + h];
                        const unsigned slot = base + static_cast<unsigned>(k + h);
                        if (slot < static_cast<unsigned>(kHitCap))
                            seq_entries(p.ws, b)[slot] = make_uint4(static_cast<unsigned>((e.j << 4) | e.m),
                                                                    __float_as_uint(s_h[h]), __float_as_uint(s_a[h]), 0u);
                    }
            }
    }

    // ---- 3. ticket: the last CTA of the sequence finishes it -----------------------------
    if (tid == 0) {
        __threadfence();                                          // entries before the ticket
        sh.last = atomicAdd(hdr + 1, 1u) == gridDim.x - 1;
        __threadfence();
    }
    if (tid <= PLDP_MAX_NGRAM) sh.ss.cnt[tid] = 0;
    __syncthreads();
    if (!sh.last) return;

    const bool has_a = p.A != nullptr;
    bool bad = false;                                             // a selected row outside [0, R)
    if (has_a && valid && p.row_idx)
        for (int k = tid; k < p.n_sel; k += kThreads) {
            const int r = __ldg(p.row_idx + k);
            bad |= r < 0 || r >= p.R;
        }
    const unsigned nh = __ldcg(hdr);
    bad = __syncthreads_or(bad) != 0;

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
            hdr[0] = 0u;
            hdr[1] = 0u;
        }
        return;
    }

    int32_t* cand_row = p.cand_pos + static_cast<int64_t>(b) * p.C_cap;
    float* hsc = (HAS_H && p.h_scores) ? p.h_scores + static_cast<int64_t>(b) * p.C_cap : nullptr;
    float* asc = (has_a && p.a_scores) ? p.a_scores + static_cast<int64_t>(b) * p.C_cap : nullptr;
    unsigned long long hk = 0, ak = 0;                            // this thread's best keys
    int nstar, total;
    if (nh <= static_cast<unsigned>(kHitCap)) {
        // ---- the list: one entry per thread ----
        const bool have = tid < static_cast<int>(nh);
        uint4 e = make_uint4(0u, 0u, 0u, 0u);
        if (have) e = __ldcg(seq_entries(p.ws, b) + tid);
        const int m = have ? static_cast<int>(e.x & 15u) : 0;
        const int32_t j = static_cast<int32_t>(e.x >> 4);
        const int wm = __reduce_max_sync(0xFFFFFFFFu, m);
        if (lane == 0) sh.wmax[warp] = wm;
        __syncthreads();
        int mx = 0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) mx = max(mx, sh.wmax[w]);
        nstar = mx >= p.ngram_min ? mx : 0;                       // m <= ngram_max already
        const bool cand = have && nstar > 0 && m >= nstar;
        sh.jl[tid] = cand ? j : INT_MAX;
        total = __syncthreads_count(cand);
        if (cand) {
            int r = 0;                                            // positions are distinct: so are ranks
            for (int k = 0; k < static_cast<int>(nh); ++k) r += sh.jl[k] < j ? 1 : 0;
            if (r < p.C_cap) {
                cand_row[r] = j;
                const float s_h = __uint_as_float(e.y), s_a = __uint_as_float(e.z);
                if (HAS_H) {
                    if (hsc) hsc[r] = s_h;
                    if (j >= 1 && s_h > p.threshold) hk = pack_key(s_h, static_cast<uint32_t>(j));
                }
                if (has_a) {
                    if (asc) asc[r] = s_a;
                    ak = pack_key(s_a, static_cast<uint32_t>(j));
                }
            }
        }
    } else {
        finish_overflow<TH, IVEC, kScoreBatch>(p, b, t, row, cand_row, hsc, asc, sh, hk, ak, nstar, total);
    }

    // ---- best of each ranking, then the draft (Sec. 4.3) ----------------------------------
    hk = warp_max_u64(hk);
    ak = warp_max_u64(ak);
    if (lane == 0) {
        sh.wkey[0][warp] = hk;
        sh.wkey[1][warp] = ak;
    }
    __syncthreads();
    if (warp != 0) return;
    hk = 0;
    ak = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
        hk = sh.wkey[0][w] > hk ? sh.wkey[0][w] : hk;
        ak = sh.wkey[1][w] > ak ? sh.wkey[1][w] : ak;
    }
    const int32_t bh = hk == 0 ? -1 : static_cast<int32_t>(key_index(hk));
    const int32_t ba = ak == 0 ? -1 : static_cast<int32_t>(key_index(ak));
    const int64_t js = p.draft_from == 0 ? bh : ba;
    int64_t dl = 0;
    if (js >= 0 && js < t) dl = (t - js < p.K) ? (t - js) : p.K;
    for (int i = lane; i < p.K; i += 32)
        p.draft[static_cast<int64_t>(b) * p.K + i] = (i < dl) ? __ldg(row + js + 1 + i) : -1;
    if (lane == 0) {
        p.cand_count[b] = total;
        p.match_len[b] = nstar;
        if (HAS_H) {
            p.best_h[b] = bh;
            if (p.best_h_score) p.best_h_score[b] = bh >= 0 ? key_value(hk) : -INFINITY;
        }
        if (has_a) {
            p.best_a[b] = ba;
            if (p.best_a_score) p.best_a_score[b] = ba >= 0 ? key_value(ak) : -INFINITY;
        }
        p.draft_len[b] = static_cast<int32_t>(dl);
        if (p.status && total > p.C_cap) atomicOr(p.status + b, PLDP_ST_CAND_OVERFLOW);
        if (p.status && bad) atomicOr(p.status + b, PLDP_ST_ROW_INDEX);
        hdr[0] = 0u;                                              // ready for the next call
        hdr[1] = 0u;
    }
}

// ---------------------------------------------------------------------------
// The incremental token index: drafting without rescanning the context.
//
// Per sequence b and token v the index holds one 64-byte entry (half a line): how
// often v occurs among the indexed positions, then up to kIndexSlots of those
// positions (in no particular order); ilen[b] is the number of positions indexed
// (0 .. ilen-1), -1 when the index of b is unusable.  A step with t = seq_len - 1:
//  * reads x_t's entry in one request (a word per lane); when the count is at
//    most kIndexSlots the slots are every occurrence before ilen, and the
//    positions appended since (ilen .. t-1, read anyway) supply the rest;
//  * otherwise (a frequent token, a stale or unusable index) falls back to the
//    ordered rescan of the context, so results are those of the scan either way;
//  * appends positions ilen .. t-1 to the index and sets ilen = t.  Each
//    appended position takes its slot with an atomic on its token's count; the
//    answer is used (the slot written) only at the end of the CTA, and tokens
//    equal to x_t take theirs only after x_t's entry has been read.
// With at most kSpeculate occurrences (most steps) every occurrence is scored
// while its suffix-match length is found, in one round trip to memory: its
// preceding tokens, the K tokens after it, H_{j-1} and the attention values at
// j are loaded together, and n* then picks the candidates among the scored
// occurrences.  With more, scoring all of them would cost more than it saves
// (each needs a d-element row and R scattered attention values): the suffix
// matches come first, then only the candidates are scored, with the tokens
// after them read in the same round trip.  One CTA per sequence.
// ---------------------------------------------------------------------------
constexpr int kIndexSlots = 15;
constexpr int kEntryWords = 1 + kIndexSlots;       // count, then the slots: 64 bytes, half a line
constexpr int kNewCap = kThreads;                  // appended positions taken in one step
constexpr int kOccCap = kIndexSlots + kNewCap;
constexpr int kDraftWin = 32;                      // draft tokens staged per occurrence (a lane each)

static_assert(kEntryWords * 4 == 64 && kEntryWords <= 32, "an entry is 64 bytes, a word per lane");

struct IndexView {
    int32_t* ilen;      // [B]
    int32_t* flags;     // [B], build scratch
    int32_t* entries;   // [B][V][kEntryWords]
    int V;
};

struct IndexShared {
    int32_t occ[kOccCap];              // occurrences of x_t, ascending
    int32_t occ_m[kOccCap];            // their suffix-match lengths
    int32_t cand[kOccCap];             // the candidates (match length >= n*), ascending
    int32_t newtok[kNewCap];           // ids of positions il .. t-1
    int32_t occ_new[kNewCap];          // the appended occurrences, ascending
    int32_t suf[PLDP_MAX_NGRAM];       // x_t, x_{t-1}, ...
    int nocc, ncand, nstar, bad_token, indexed, wmax[kWarps];
};

__device__ __forceinline__ int32_t* index_entry(const IndexView& ix, int b, int32_t tok) {
    return ix.entries + (static_cast<int64_t>(b) * ix.V + tok) * kEntryWords;
}

// Counts one more occurrence of token tok in sequence b's index: returns the slot
// it takes (the old count; >= kIndexSlots: none), or -1 for a token outside [0, V).
__device__ __forceinline__ int index_take(const IndexView& ix, int b, int32_t tok) {
    if (tok < 0 || tok >= ix.V) return -1;
    return atomicAdd(index_entry(ix, b, tok), 1);
}

// Writes position q into the slot taken by index_take.
__device__ __forceinline__ void index_put(const IndexView& ix, int b, int32_t tok, int slot, int64_t q) {
    if (slot >= 0 && slot < kIndexSlots) index_entry(ix, b, tok)[1 + slot] = static_cast<int32_t>(q);
}

__device__ __forceinline__ bool index_insert(const IndexView& ix, int b, int64_t q, int32_t tok) {
    const int slot = index_take(ix, b, tok);
    index_put(ix, b, tok, slot, q);
    return slot >= 0;
}

// The indexed drafting of sequence b by the whole CTA, for context length L.
// RD: how ids are read -- CoherentIds when this kernel has just appended to the
// context (verification fused in front), else through the read-only cache.
// PRE: the indexed length is il_in and the ids it starts from -- is.newtok (the
// positions appended since, when they fit) and is.suf (x_t, x_{t-1}, ...) -- are
// already in shared memory, written before the CTA's last barrier.
template <typename TH, bool IVEC, typename RD, bool PRE = false>
__device__ __forceinline__ void index_draft(const DraftParams& p, const IndexView& ix, int b, int64_t L,
                                            StepShared& sh, IndexShared& is, int64_t il_in = 0) {
    constexpr bool HAS_H = !std::is_same<TH, NoHidden>::value;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t il = PRE ? il_in : static_cast<int64_t>(ix.ilen[b]);
    const bool valid = L >= 0 && L <= p.T_cap;
    const int64_t t = L - 1;
    const int32_t* row = p.ids + static_cast<int64_t>(b) * p.ids_stride;
    const bool has_a = p.A != nullptr;
    const size_t h_es = p.h_bf16 ? 2 : 4;
    bool bad = false;                                             // a selected row outside [0, R)
    if (has_a && valid && p.row_idx)
        for (int k = tid; k < p.n_sel; k += kThreads) {
            const int r = __ldg(p.row_idx + k);
            bad |= r < 0 || r >= p.R;
        }
    if (tid <= PLDP_MAX_NGRAM) sh.ss.cnt[tid] = 0;
    if (tid == 0) is.bad_token = 0;
    bad = __syncthreads_or(bad) != 0;
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
    // usable: the index covers a prefix of the context; small: what was appended fits the CTA
    const bool usable = il >= 0 && il <= t;
    const int64_t nnew = usable ? t - il : 0;
    const bool small = usable && nnew <= kNewCap;
    if (tid == 0 && HAS_H && t >= 2)                              // H_{t-1}: every candidate's score reads it
        prefetch_l2_bulk(static_cast<const char*>(p.H) + (static_cast<int64_t>(b) * p.h_seq_stride + (t - 1) * p.d) * h_es,
                         static_cast<uint32_t>(p.d * h_es));
    if (!PRE) {
        if (small && tid < nnew) is.newtok[tid] = RD::one(row + il + tid);
        if (tid < PLDP_MAX_NGRAM) is.suf[tid] = (tid < p.ngram_max && t - tid >= 0) ? RD::one(row + t - tid) : 0;
    }
    __syncthreads();
    const int32_t xt = is.suf[0];
    const bool lookup = small && t >= 1 && xt >= 0 && xt < ix.V;
    int32_t ev = 0;                                               // x_t's entry, word `lane` (warp 0)
    if (lookup && tid < kEntryWords) ev = __ldcg(index_entry(ix, b, xt) + tid);
    // this thread's appended position (small): its token and the slot it takes
    const bool mine = small && tid < nnew;
    const int32_t mytok = mine ? is.newtok[tid] : 0;
    int myslot = -1;
    if (mine && mytok != xt) myslot = index_take(ix, b, mytok);  // other entries: no wait for x_t's
    if (mine && (mytok < 0 || mytok >= ix.V)) atomicOr(&is.bad_token, 1);
    if (warp == 0 && lookup) {
        // the appended occurrences (ascending) while the entry is on its way
        int nn = 0;
        for (int c0 = 0; c0 < nnew; c0 += 32) {
            const bool hit = c0 + lane < nnew && is.newtok[c0 + lane] == xt;
            const unsigned bal = __ballot_sync(0xFFFFFFFFu, hit);
            if (hit) is.occ_new[nn + __popc(bal & ((1u << lane) - 1u))] = static_cast<int32_t>(il + c0 + lane);
            nn += __popc(bal);
        }
        const int nold = __shfl_sync(0xFFFFFFFFu, ev, 0);
        const bool ok = nold >= 0 && nold <= kIndexSlots;         // else the slots do not hold them all
        if (ok) {
            if (lane >= 1 && lane <= nold) {                      // the indexed ones (all before il), ranked
                int rank = 0;
                for (int k = 1; k <= nold; ++k) rank += __shfl_sync((1u << (nold + 1)) - 2u, ev, k) < ev ? 1 : 0;
                is.occ[rank] = ev;
            }
            __syncwarp();
            for (int k = lane; k < nn; k += 32) is.occ[nold + k] = is.occ_new[k];
        }
        if (lane == 0) {
            is.indexed = ok;
            is.nocc = ok ? nold + nn : 0;
        }
    }
    __syncthreads();                                              // x_t's entry has been read
    const bool indexed = lookup && is.indexed;
    if (mine && mytok == xt) myslot = index_take(ix, b, mytok);
    if (usable && !small) {                                       // a long append: inserted in turn
        bool badtok = false;
        for (int64_t q = il + tid; q < t; q += kThreads) badtok |= !index_insert(ix, b, q, RD::one(row + q));
        if (badtok) atomicOr(&is.bad_token, 1);
    }

    int32_t* cand_row = p.cand_pos + static_cast<int64_t>(b) * p.C_cap;
    float* hsc = (HAS_H && p.h_scores) ? p.h_scores + static_cast<int64_t>(b) * p.C_cap : nullptr;
    float* asc = (has_a && p.a_scores) ? p.a_scores + static_cast<int64_t>(b) * p.C_cap : nullptr;
    const int nocc = indexed ? is.nocc : 0;
    // More occurrences than are scored at once: the suffix matches come first, and
    // meanwhile the rows of (up to kPrefetchOcc of) the occurrences head for L2 --
    // H_{j-1} with one bulk prefetch, the attention values at key j when the
    // selected rows of a key are side by side -- so that the candidates' scoring,
    // a round trip later, finds them there.
    if (indexed && nocc > kSpeculate && tid < nocc && tid < kPrefetchOcc) {
        const int64_t j = is.occ[tid];
        if (HAS_H && j >= 1 && j < t)
            prefetch_l2_bulk(static_cast<const char*>(p.H) + (static_cast<int64_t>(b) * p.h_seq_stride + (j - 1) * p.d) * h_es,
                             static_cast<uint32_t>(p.d * h_es));
        if (has_a && p.a_row_stride == 1 && !p.row_idx && j >= 0 && j < t) {
            const size_t a_es = p.a_bf16 ? 2 : 4;
            const char* run = static_cast<const char*>(p.A) + (static_cast<int64_t>(b) * p.a_seq_stride + j * p.a_key_stride) * a_es;
            const char* end = run + static_cast<int64_t>(p.R) * a_es;          // every address inside the run
            for (const char* a = run; a < end; a += 128) asm volatile("prefetch.global.L2 [%0];" ::"l"(a));
            asm volatile("prefetch.global.L2 [%0];" ::"l"(end - 1));
        }
    }

    // Warp 0: the choices of both rankings (best keys hk, ak), the draft (Sec. 4.3)
    // with draft_tok(i, j*) giving token j* + 1 + i, and the per-sequence outputs.
    auto outputs = [&](unsigned long long hk, unsigned long long ak, int nstar, int total, auto draft_tok) {
        const int32_t bh = hk == 0 ? -1 : static_cast<int32_t>(key_index(hk));
        const int32_t ba = ak == 0 ? -1 : static_cast<int32_t>(key_index(ak));
        const int64_t js = p.draft_from == 0 ? bh : ba;
        int64_t dl = 0;
        if (js >= 0 && js < t) dl = (t - js < p.K) ? (t - js) : p.K;
        for (int i = lane; i < p.K; i += 32)
            p.draft[static_cast<int64_t>(b) * p.K + i] = (i < dl) ? draft_tok(i, js) : -1;
        if (lane == 0) {
            p.cand_count[b] = total;
            p.match_len[b] = nstar;
            if (HAS_H) {
                p.best_h[b] = bh;
                if (p.best_h_score) p.best_h_score[b] = bh >= 0 ? key_value(hk) : -INFINITY;
            }
            if (has_a) {
                p.best_a[b] = ba;
                if (p.best_a_score) p.best_a_score[b] = ba >= 0 ? key_value(ak) : -INFINITY;
            }
            p.draft_len[b] = static_cast<int32_t>(dl);
            if (p.status && total > p.C_cap) atomicOr(p.status + b, PLDP_ST_CAND_OVERFLOW);
            if (p.status && bad) atomicOr(p.status + b, PLDP_ST_ROW_INDEX);
            // the index now covers 0 .. t-1 (or is unusable: a token it cannot hold, or stale)
            if (usable) ix.ilen[b] = is.bad_token ? -1 : static_cast<int32_t>(t);
            else if (il > t && il > 0) ix.ilen[b] = -1;         // shrunk (an empty context keeps il = 0)
        }
    };

    // ---- the list scored: every occurrence, or the candidates --------------------------
    // spec: at most kSpeculate occurrences, all scored at once; their suffix matches
    // are read in the same round trip and n* then picks the candidates among them.
    // Otherwise the suffix matches come first (each scored occurrence costs a
    // d-element row and R scattered attention values) and only the candidates
    // (the first C_cap) are scored.  Either way one loop with one call of the
    // scorer, kSpeculate positions a pass: every case runs the same code.
    constexpr int NB = kSpeculate;
    unsigned long long hk = 0, ak = 0;
    int nstar = 0, total = 0;
    const bool spec = indexed && nocc <= kSpeculate;
    if (indexed && !spec) {
        int mloc = 0;
        for (int i = tid; i < nocc; i += kThreads) {
            const int64_t j = is.occ[i];
            int32_t pv[PLDP_MAX_NGRAM - 1];                       // x_{j-1}, x_{j-2}, ... all requested at once
#pragma unroll
            for (int m = 1; m < PLDP_MAX_NGRAM; ++m) {
                const int64_t q = j - m;
                pv[m - 1] = (m < p.ngram_max && q >= 0) ? (q >= il ? is.newtok[q - il] : RD::one(row + q)) : 0;
            }
            int m = 1;
#pragma unroll
            for (int k = 1; k < PLDP_MAX_NGRAM; ++k)
                if (m == k && k < p.ngram_max && j - k >= 0 && pv[k - 1] == is.suf[k]) m = k + 1;
            is.occ_m[i] = m;
            mloc = m > mloc ? m : mloc;
        }
        mloc = __reduce_max_sync(0xFFFFFFFFu, mloc);
        if (lane == 0) is.wmax[warp] = mloc;
        __syncthreads();
        if (warp == 0) {
            int mx = 0;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) mx = is.wmax[w] > mx ? is.wmax[w] : mx;
            const int ns = mx >= p.ngram_min ? mx : 0;           // m <= ngram_max already
            int base = 0;
            if (ns > 0)
                for (int c0 = 0; c0 < nocc; c0 += 32) {
                    const bool c = c0 + lane < nocc && is.occ_m[c0 + lane] >= ns;
                    const unsigned bal = __ballot_sync(0xFFFFFFFFu, c);
                    if (c) {
                        const int r = base + __popc(bal & ((1u << lane) - 1u));
                        is.cand[r] = is.occ[c0 + lane];
                        if (r < p.C_cap) cand_row[r] = is.occ[c0 + lane];
                    }
                    base += __popc(bal);
                }
            if (lane == 0) {
                is.nstar = ns;
                is.ncand = base;
            }
        }
        __syncthreads();
        nstar = is.nstar;
        total = is.ncand;
    } else if (!indexed) {
        finish_overflow<TH, IVEC, kMaxScoreBatch, RD>(p, b, t, row, cand_row, hsc, asc, sh, hk, ak, nstar, total);
    }

    if (indexed) {
        const int32_t* list = spec ? is.occ : is.cand;
        const int n = spec ? nocc : (total < p.C_cap ? total : p.C_cap);
        int32_t pre[PLDP_MAX_NGRAM - 1];                          // spec, thread h < n: x_{j-1}, x_{j-2}, ...
        const int64_t jm = (spec && tid < n) ? list[tid] : -1;
#pragma unroll
        for (int m = 1; m < PLDP_MAX_NGRAM; ++m) {
            const int64_t q = jm - m;
            pre[m - 1] = (jm >= 0 && m < p.ngram_max && q >= 0) ? (q >= il ? is.newtok[q - il] : RD::one(row + q)) : 0;
        }
        const bool staged = p.K <= kDraftWin;                     // warp 0, lane i: token i after list[h], h < NB
        int32_t dv[NB];
        int64_t j0[NB];
#pragma unroll
        for (int h = 0; h < NB; ++h) {
            j0[h] = h < n ? list[h] : -1;
            const int64_t q = j0[h] + 1 + lane;
            dv[h] = (staged && warp == 0 && h < n && lane < p.K && q <= t) ? RD::one(row + q) : -1;
        }
        float s_h[NB], s_a[NB];
        for (int i0 = 0; i0 < n; i0 += NB) {                      // one pass but for many candidates
            const int nb = n - i0 < NB ? n - i0 : NB;
            int64_t j[NB];
#pragma unroll
            for (int h = 0; h < NB; ++h) j[h] = h < nb ? list[i0 + h] : -1;
            cta_score<TH, NB>(p, b, j, nb, t, part_buf<NB>(sh.part[(i0 / NB) & 1]), s_h, s_a);
            if (!spec && warp == 0)                               // candidates: keys now
#pragma unroll
                for (int h = 0; h < NB; ++h) {
                    if (h >= nb) continue;
                    const int r = i0 + h;
                    if (HAS_H) {
                        if (hsc && lane == 0) hsc[r] = s_h[h];
                        if (j[h] >= 1 && s_h[h] > p.threshold) {
                            const unsigned long long key = pack_key(s_h[h], static_cast<uint32_t>(j[h]));
                            hk = key > hk ? key : hk;
                        }
                    }
                    if (has_a) {
                        if (asc && lane == 0) asc[r] = s_a[h];
                        const unsigned long long key = pack_key(s_a[h], static_cast<uint32_t>(j[h]));
                        ak = key > ak ? key : ak;
                    }
                }
        }
        if (mine) index_put(ix, b, mytok, myslot, il + tid);      // the slot taken above
        if (warp != 0) return;
        if (spec) {
            // n* among the scored occurrences (n <= NB: one pass), then their keys
            int m = 0;
            if (lane < n) {
                m = 1;
#pragma unroll
                for (int k = 1; k < PLDP_MAX_NGRAM; ++k)
                    if (m == k && k < p.ngram_max && jm - k >= 0 && pre[k - 1] == is.suf[k]) m = k + 1;
            }
            int mh[NB], mx = 0;
#pragma unroll
            for (int h = 0; h < NB; ++h) {
                mh[h] = __shfl_sync(0xFFFFFFFFu, m, h);
                mx = mh[h] > mx ? mh[h] : mx;
            }
            nstar = mx >= p.ngram_min ? mx : 0;                   // m <= ngram_max already
            int r = 0;                                            // candidates: ascending, as the occurrences
            if (nstar > 0)
#pragma unroll
                for (int h = 0; h < NB; ++h) {
                    if (h >= n || mh[h] < nstar) continue;
                    if (r < p.C_cap) {
                        if (lane == 0) cand_row[r] = static_cast<int32_t>(j0[h]);
                        if (HAS_H) {
                            if (hsc && lane == 0) hsc[r] = s_h[h];
                            if (j0[h] >= 1 && s_h[h] > p.threshold) {
                                const unsigned long long key = pack_key(s_h[h], static_cast<uint32_t>(j0[h]));
                                hk = key > hk ? key : hk;
                            }
                        }
                        if (has_a) {
                            if (asc && lane == 0) asc[r] = s_a[h];
                            const unsigned long long key = pack_key(s_a[h], static_cast<uint32_t>(j0[h]));
                            ak = key > ak ? key : ak;
                        }
                    }
                    ++r;
                }
            total = r;
        }
        outputs(hk, ak, nstar, total, [&](int i, int64_t js) -> int32_t {
            if (staged && i == lane) {
                int32_t v = -1;
                bool found = false;
#pragma unroll
                for (int h = 0; h < NB; ++h)
                    if (h < n && j0[h] == js) {
                        v = dv[h];
                        found = true;
                    }
                if (found) return v;
            }
            return RD::one(row + js + 1 + i);
        });
        return;
    }

    // ---- the rescan's keys, combined over the CTA, then the outputs ---------------------
    hk = warp_max_u64(hk);
    ak = warp_max_u64(ak);
    if (lane == 0) {
        sh.wkey[0][warp] = hk;
        sh.wkey[1][warp] = ak;
    }
    if (mine) index_put(ix, b, mytok, myslot, il + tid);          // the slot taken above
    __syncthreads();
    if (warp != 0) return;
    hk = 0;
    ak = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
        hk = sh.wkey[0][w] > hk ? sh.wkey[0][w] : hk;
        ak = sh.wkey[1][w] > ak ? sh.wkey[1][w] : ak;
    }
    outputs(hk, ak, nstar, total, [&](int i, int64_t js) -> int32_t { return RD::one(row + js + 1 + i); });
}

template <typename TH, bool IVEC>
__global__ void __launch_bounds__(kThreads, 1) draft_index_kernel(const DraftParams p, const IndexView ix) {
    __shared__ StepShared sh;
    __shared__ IndexShared is;
    pdl_enter();
    index_draft<TH, IVEC, ReadOnlyIds>(p, ix, blockIdx.x, p.seq_len[blockIdx.x], sh, is);
}

// Verification of the current step -- the finish of greedy verification: the
// accepted length, the bonus token and the append (Sec. 4.4) -- and then, in the
// same CTA, the next step's drafting with the token index.  One CTA per
// sequence, launched behind the verification's argmax pass (greedy: the targets
// are the row keys) or behind the draws of sampling verification (va.row_draws).  The draft step
// starts from the context the finish has just written: its length is known
// without a read, and the appended ids are read through L2.
constexpr int kOldWin = 32;                        // old-context tokens read before the wait (a lane each)

template <typename TH, bool IVEC>
__global__ void __launch_bounds__(kThreads, 1) verify_draft_kernel(const VerifyArgs va, const DraftParams p,
                                                                    const IndexView ix) {
    __shared__ StepShared sh;
    __shared__ IndexShared is;
    __shared__ long long L_after;
    __shared__ int32_t oldwin[kOldWin];                          // x_{Lw}, ..., x_{Lw + kOldWin - 1}
    const int b = blockIdx.x;
    // Read before the wait, since the argmax pass does not write them (its
    // predecessors, which did, completed before it started): the indexed length,
    // the last kOldWin tokens of the context as it was before this step's append --
    // the drafting's appended ids and suffix reach back into them -- and the
    // finish's draft, draft length and context length.
    const int64_t il = ix.ilen[b];
    const int64_t L_old = va.seq_len ? static_cast<int64_t>(va.seq_len[b]) : -1;
    const int64_t Lw = L_old - kOldWin;
    const int32_t* row_b = p.ids + static_cast<int64_t>(b) * p.ids_stride;
    FinishIn fin = {};
    if (threadIdx.x < kOldWin) {
        const int64_t q = Lw + threadIdx.x;
        oldwin[threadIdx.x] = (L_old >= 1 && L_old <= p.T_cap && q >= 0) ? __ldcg(row_b + q) : 0;
        fin = finish_inputs(va, b, static_cast<int>(threadIdx.x));    // the draft: not written by the pass
    }
    pdl_enter();                                                  // the pass's row keys are final
    if (threadIdx.x < 32) {
        const int lane = static_cast<int>(threadIdx.x);
        __syncwarp();                                             // oldwin written by this warp
        FinishOut fo;
        const int64_t r0 = static_cast<int64_t>(b) * (va.K + 1);
        const RowTokens src{va.row_draws ? nullptr : va.row_keys + r0, va.row_draws ? va.row_draws + r0 : nullptr};
        const int64_t L1 = finish_sequence(va, b, lane, src, &fo, &fin);
        if (lane == 0) L_after = L1;
        // The drafting's first reads come from what the finish holds: the ids appended
        // since the index was brought up to date (il .. t-1) and the suffix x_t, x_{t-1},
        // ...; positions the finish wrote come from its draft and bonus, older ones from L2.
        if (L1 >= 0 && L1 <= p.T_cap) {
            const int64_t t = L1 - 1;
            const int64_t L0 = fo.appended ? L1 - fo.n - 1 : L1;  // the first appended position
            const int32_t* row = p.ids + static_cast<int64_t>(b) * p.ids_stride;
            const int32_t* dr = va.draft + static_cast<int64_t>(b) * va.K;
            auto tok = [&](int64_t q) -> int32_t {
                if (q >= L0) return q - L0 < fo.n ? dr[q - L0] : fo.bonus;
                if (L0 == L_old && q >= Lw) return oldwin[q - Lw];     // read before the wait
                return __ldcg(row + q);
            };
            const bool usable = il >= 0 && il <= t;
            const int64_t nnew = usable ? t - il : 0;
            if (usable && nnew <= kNewCap)
                for (int64_t k = lane; k < nnew; k += 32) is.newtok[k] = tok(il + k);
            if (lane < PLDP_MAX_NGRAM) is.suf[lane] = (lane < p.ngram_max && t - lane >= 0) ? tok(t - lane) : 0;
        } else if (lane < PLDP_MAX_NGRAM) {
            is.suf[lane] = 0;                                     // no last token (as the drafting reads it)
        }
    }
    __syncthreads();                                              // the append is visible to the whole CTA
    const int64_t L = L_after >= 0 ? static_cast<int64_t>(L_after) : static_cast<int64_t>(__ldcg(p.seq_len + b));
    index_draft<TH, IVEC, CoherentIds, true>(p, ix, b, L, sh, is, il);
}

// Index build: positions 0 .. seq_len-2 of every sequence.
__global__ void __launch_bounds__(kThreads) index_build_kernel(const int32_t* __restrict__ ids, int64_t ids_stride,
                                                               const int32_t* __restrict__ seq_len, int64_t T_cap,
                                                               IndexView ix) {
    pdl_enter();
    const int b = blockIdx.y;
    const int64_t L = seq_len[b];
    if (L < 0 || L > T_cap) return;
    const int64_t t = L - 1;
    const int32_t* row = ids + static_cast<int64_t>(b) * ids_stride;
    for (int64_t q = static_cast<int64_t>(blockIdx.x) * kThreads + threadIdx.x; q < t;
         q += static_cast<int64_t>(gridDim.x) * kThreads)
        if (!index_insert(ix, b, q, __ldg(row + q))) atomicOr(ix.flags + b, 1);
}

__global__ void index_finish_kernel(const int32_t* __restrict__ seq_len, int B, int64_t T_cap, IndexView ix,
                                    uint32_t* __restrict__ status) {
    pdl_enter();
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= B) return;
    const int64_t L = seq_len[b];
    if (L < 0 || L > T_cap) {
        ix.ilen[b] = -1;
        if (status) atomicOr(status + b, PLDP_ST_SEQ_LEN);
        return;
    }
    const bool bad_token = ix.flags[b] != 0;
    ix.ilen[b] = bad_token ? -1 : static_cast<int32_t>(L >= 1 ? L - 1 : 0);
    if (bad_token && status) atomicOr(status + b, PLDP_ST_TOKEN_RANGE);
}

// Byte offsets of the index parts (ilen, flags, entries), 256-byte aligned.
struct IndexLayout {
    size_t ilen, flags, entries, total;
};
inline IndexLayout index_layout(int B, int V) {
    auto up = [](size_t x) { return (x + 255) / 256 * 256; };
    IndexLayout l;
    l.ilen = 0;
    l.flags = up(static_cast<size_t>(B) * 4);
    l.entries = l.flags + up(static_cast<size_t>(B) * 4);
    l.total = l.entries + up(static_cast<size_t>(B) * V * kEntryWords * 4);
    return l;
}
inline IndexView index_view(void* base, int B, int V) {
    const IndexLayout l = index_layout(B, V);
    char* c = static_cast<char*>(base);
    return IndexView{reinterpret_cast<int32_t*>(c + l.ilen), reinterpret_cast<int32_t*>(c + l.flags),
                     reinterpret_cast<int32_t*>(c + l.entries), V};
}

template <typename TH, bool IVEC>
pldp_status launch_t(const DraftParams& p, int B, cudaStream_t s) {
    int64_t chunks = (p.T_cap + kChunk - 1) / kChunk;
    if (chunks < 1) chunks = 1;                                   // every sequence needs its finish
    if (chunks > 65535) return fail(PLDP_ERR_UNSUPPORTED, "draft_step: T_cap too large for the grid");
    cudaError_t e = launch_pdl(draft_step_kernel<TH, IVEC>,
                               dim3(static_cast<unsigned>(chunks), static_cast<unsigned>(B)), dim3(kThreads), 0, s,
                               0, p);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "draft_step: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}

template <typename TH, bool IVEC>
pldp_status launch_index_t(const DraftParams& p, const IndexView& ix, int B, cudaStream_t s) {
    cudaError_t e = launch_pdl(draft_index_kernel<TH, IVEC>, dim3(static_cast<unsigned>(B)), dim3(kThreads), 0, s, 0,
                               p, ix);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "draft_step (indexed): launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}

template <typename TH>
pldp_status launch_draft_step(const DraftParams& p, int B, cudaStream_t s, bool ivec, const IndexView* ix) {
    if (ix) return ivec ? launch_index_t<TH, true>(p, *ix, B, s) : launch_index_t<TH, false>(p, *ix, B, s);
    return ivec ? launch_t<TH, true>(p, B, s) : launch_t<TH, false>(p, B, s);
}

// The checks and argument block of pldp_draft_step (`what` names the call in
// messages).  empty: B == 0, nothing to launch.
pldp_status prepare_draft(const pldp_draft_step_args* a, const char* what, DraftParams& p, IndexView& ixv,
                          bool& has_ix, bool& ivec, bool& empty) {
    const int B = a->B;
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "%s: B < 0", what);
    if (B > 65535) return fail(PLDP_ERR_UNSUPPORTED, "%s: B > 65535", what);
    if (a->T_cap < 0 || a->T_cap > kMaxPositions)
        return fail(PLDP_ERR_INVALID_ARG, "%s: T_cap outside [0, 2^27]", what);
    if (a->ids_stride < a->T_cap) return fail(PLDP_ERR_INVALID_ARG, "%s: ids_stride < T_cap", what);
    if (a->ngram_min < 1 || a->ngram_max < a->ngram_min || a->ngram_max > PLDP_MAX_NGRAM)
        return fail(PLDP_ERR_INVALID_ARG, "%s: need 1 <= ngram_min <= ngram_max <= %d", what,
                    PLDP_MAX_NGRAM);
    if (a->C_cap < 0) return fail(PLDP_ERR_INVALID_ARG, "%s: C_cap < 0", what);
    if (a->K < 1) return fail(PLDP_ERR_INVALID_ARG, "%s: K < 1", what);
    if (!a->H && !a->A) return fail(PLDP_ERR_INVALID_ARG, "%s: neither H nor A given", what);
    if (a->draft_from != 0 && a->draft_from != 1)
        return fail(PLDP_ERR_INVALID_ARG, "%s: draft_from must be 0 (hidden) or 1 (attention)", what);
    if ((a->draft_from == 0 && !a->H) || (a->draft_from == 1 && !a->A))
        return fail(PLDP_ERR_INVALID_ARG, "%s: draft_from names a ranking that is not given", what);
    size_t qbytes = 0, h_es = 0;
    if (a->H) {
        if (a->h_dtype != PLDP_F32 && a->h_dtype != PLDP_BF16)
            return fail(PLDP_ERR_UNSUPPORTED, "%s: unsupported hidden dtype %d", what, (int)a->h_dtype);
        h_es = a->h_dtype == PLDP_F32 ? 4 : 2;
        if (a->d < 1) return fail(PLDP_ERR_INVALID_ARG, "%s: d < 1", what);
        qbytes = static_cast<size_t>(a->d) * h_es;
        if (qbytes > kMaxQueryBytes)
            return fail(PLDP_ERR_UNSUPPORTED, "%s: d * sizeof(dtype) > %zu", what, kMaxQueryBytes);
        if (a->h_seq_stride < a->T_cap * a->d)
            return fail(PLDP_ERR_INVALID_ARG, "%s: h_seq_stride < T_cap*d", what);
        if (a->threshold != a->threshold) return fail(PLDP_ERR_INVALID_ARG, "%s: threshold is NaN", what);
    }
    int sel = 0;
    if (a->A) {
        if (a->a_dtype != PLDP_F32 && a->a_dtype != PLDP_BF16)
            return fail(PLDP_ERR_UNSUPPORTED, "%s: unsupported attention dtype %d", what, (int)a->a_dtype);
        if (a->agg != PLDP_AGG_MAX && a->agg != PLDP_AGG_SUM)
            return fail(PLDP_ERR_INVALID_ARG, "%s: unknown aggregation %d", what, (int)a->agg);
        if (a->R < 1) return fail(PLDP_ERR_INVALID_ARG, "%s: R < 1", what);
        if (const char* why = attention_layout_error(a->R, a->T_cap, a->a_row_stride,
                                                     a->a_key_stride == 0 ? 1 : a->a_key_stride, a->a_seq_stride))
            return fail(PLDP_ERR_INVALID_ARG, "%s: attention layout: %s", what, why);
        sel = a->row_idx ? a->n_sel : a->R;
        if (sel < 1 || sel > kMaxSelRows)
            return fail(PLDP_ERR_INVALID_ARG, "%s: need 1 <= n_sel <= %d", what, kMaxSelRows);
    }
    empty = B == 0;
    if (empty) return PLDP_OK;
    if (!a->ids || !a->seq_len || !a->cand_count || !a->match_len || !a->draft || !a->draft_len ||
        (a->C_cap > 0 && !a->cand_pos) || (a->H && !a->best_h) || (a->A && !a->best_a))
        return fail(PLDP_ERR_INVALID_ARG, "%s: null pointer", what);
    has_ix = a->index != nullptr;
    if (a->index) {
        if (a->V < 1) return fail(PLDP_ERR_INVALID_ARG, "%s: V < 1 with an index", what);
        const size_t need = index_layout(B, a->V).total;
        if (a->index_bytes < need || !aligned16(a->index))
            return fail(PLDP_ERR_INVALID_ARG, "%s: index needs %zu bytes, 16-byte aligned", what, need);
        ixv = index_view(a->index, B, a->V);
    } else if (!a->workspace || a->workspace_bytes < static_cast<size_t>(B) * kSeqWs || !aligned16(a->workspace)) {
        return fail(PLDP_ERR_INVALID_ARG, "%s: workspace needs %zu bytes, 16-byte aligned", what,
                    static_cast<size_t>(B) * kSeqWs);
    }
    if (a->H && !(aligned16(a->H) && qbytes % 16 == 0 && (a->h_seq_stride * h_es) % 16 == 0))
        return fail(PLDP_ERR_UNSUPPORTED,
                    "draft_step: hidden rows must be 16-byte aligned (the separate calls accept any layout)");

    p = DraftParams{};
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
    p.a_key_stride = a->a_key_stride == 0 ? 1 : a->a_key_stride;
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
    ivec = aligned16(a->ids) && a->ids_stride % 4 == 0 && a->T_cap % 4 == 0;
    return PLDP_OK;
}

template <typename TH, bool IVEC>
pldp_status launch_verify_draft_t(const VerifyArgs& va, const DraftParams& p, const IndexView& ix, int B,
                                  cudaStream_t s) {
    const cudaError_t e = launch_pdl(verify_draft_kernel<TH, IVEC>, dim3(static_cast<unsigned>(B)), dim3(kThreads), 0,
                                     s, 0, va, p, ix);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "verify_draft: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}

template <typename TH>
pldp_status launch_verify_draft(const VerifyArgs& va, const DraftParams& p, const IndexView& ix, int B, bool ivec,
                                cudaStream_t s) {
    return ivec ? launch_verify_draft_t<TH, true>(va, p, ix, B, s) : launch_verify_draft_t<TH, false>(va, p, ix, B, s);
}

}  // namespace
}  // namespace pldp

using namespace pldp;

extern "C" PLDP_API size_t pldp_draft_workspace_size(int B) {
    return B < 0 ? 0 : static_cast<size_t>(B) * kSeqWs;
}

extern "C" PLDP_API pldp_status pldp_draft_step(const pldp_draft_step_args* a, void* stream) {
    if (!a) return fail(PLDP_ERR_INVALID_ARG, "draft_step: null argument block");
    DraftParams p;
    IndexView ixv = {};
    bool has_ix = false, ivec = false, empty = false;
    const pldp_status st = prepare_draft(a, "draft_step", p, ixv, has_ix, ivec, empty);
    if (st != PLDP_OK || empty) return st;
    const int B = a->B;
    const IndexView* ix = has_ix ? &ixv : nullptr;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (!a->H) return launch_draft_step<NoHidden>(p, B, s, ivec, ix);
    if (a->h_dtype == PLDP_BF16) return launch_draft_step<__nv_bfloat16>(p, B, s, ivec, ix);
    return launch_draft_step<float>(p, B, s, ivec, ix);
}

extern "C" PLDP_API pldp_status pldp_verify_greedy_draft(const pldp_verify_draft_args* a, void* stream) {
    if (!a) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_draft: null argument block");
    const pldp_draft_step_args& n = a->next;
    if (!n.index) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_draft: the next draft needs a token index");
    if (a->V < 1) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_draft: V < 1");
    if (n.V != a->V) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_draft: the index's V differs from the logits'");
    if (a->dtype != PLDP_F32 && a->dtype != PLDP_BF16)
        return fail(PLDP_ERR_UNSUPPORTED, "verify_greedy_draft: unsupported dtype %d", (int)a->dtype);
    if (n.T_cap > INT32_MAX) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_draft: bad T_cap");
    DraftParams p;
    IndexView ixv = {};
    bool has_ix = false, ivec = false, empty = false;
    const pldp_status st = prepare_draft(&n, "verify_greedy_draft", p, ixv, has_ix, ivec, empty);
    if (st != PLDP_OK || empty) return st;
    const int B = n.B, K = n.K;
    if (!a->logits || !a->draft || !a->draft_len || !a->accept_len || !a->next_token)
        return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_draft: null pointer");
    const size_t need = pldp_verify_workspace_size(B, K, a->V);
    if (!a->workspace || a->workspace_bytes < need || !aligned16(a->workspace))
        return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_draft: workspace needs %zu bytes, 16-byte aligned", need);
    // verification appends to the context the next draft reads: next.ids and next.seq_len
    VerifyArgs va = verify_args(B, K, a->V, a->draft, a->draft_len, a->argmax, a->accept_len, a->next_token,
                                const_cast<int32_t*>(n.ids), n.ids_stride, const_cast<int32_t*>(n.seq_len), n.T_cap,
                                a->kv_keep_len, n.status);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const pldp_status sp = launch_verify_pass(a->logits, a->dtype, va, a->workspace, s, "verify_greedy_draft");
    if (sp != PLDP_OK) return sp;
    if (!n.H) return launch_verify_draft<NoHidden>(va, p, ixv, B, ivec, s);
    if (n.h_dtype == PLDP_BF16) return launch_verify_draft<__nv_bfloat16>(va, p, ixv, B, ivec, s);
    return launch_verify_draft<float>(va, p, ixv, B, ivec, s);
}

extern "C" PLDP_API size_t pldp_verify_sample_draft_workspace_size(int B, int K, int V, pldp_dtype dtype) {
    return sample_draft_workspace_size(B, K, V, dtype);
}

extern "C" PLDP_API pldp_status pldp_verify_sample_draft(const pldp_verify_sample_draft_args* a, void* stream) {
    if (!a) return fail(PLDP_ERR_INVALID_ARG, "verify_sample_draft: null argument block");
    const pldp_draft_step_args& n = a->next;
    if (!n.index) return fail(PLDP_ERR_INVALID_ARG, "verify_sample_draft: the next draft needs a token index");
    if (a->V < 1) return fail(PLDP_ERR_INVALID_ARG, "verify_sample_draft: V < 1");
    if (n.V != a->V) return fail(PLDP_ERR_INVALID_ARG, "verify_sample_draft: the index's V differs from the logits'");
    if (a->dtype != PLDP_F32 && a->dtype != PLDP_BF16)
        return fail(PLDP_ERR_UNSUPPORTED, "verify_sample_draft: unsupported dtype %d", (int)a->dtype);
    if (!(a->temperature > 0.f) || isinf(a->temperature))
        return fail(PLDP_ERR_INVALID_ARG, "verify_sample_draft: temperature must be positive and finite");
    if (n.T_cap > INT32_MAX) return fail(PLDP_ERR_INVALID_ARG, "verify_sample_draft: bad T_cap");
    if (n.K >= 1 && static_cast<int64_t>(n.K) + 1 > 12288)
        return fail(PLDP_ERR_UNSUPPORTED, "verify_sample_draft: K > 12287");
    DraftParams p;
    IndexView ixv = {};
    bool has_ix = false, ivec = false, empty = false;
    const pldp_status st = prepare_draft(&n, "verify_sample_draft", p, ixv, has_ix, ivec, empty);
    if (st != PLDP_OK || empty) return st;
    const int B = n.B, K = n.K;
    if (!a->logits || !a->uniforms || !a->draft || !a->draft_len || !a->accept_len || !a->next_token)
        return fail(PLDP_ERR_INVALID_ARG, "verify_sample_draft: null pointer");
    const size_t need = sample_draft_workspace_size(B, K, a->V, a->dtype);
    if (!a->workspace || a->workspace_bytes < need || !aligned16(a->workspace))
        return fail(PLDP_ERR_INVALID_ARG, "verify_sample_draft: workspace needs %zu bytes, 16-byte aligned", need);
    // verification appends to the context the next draft reads: next.ids and next.seq_len
    VerifyArgs va = verify_args(B, K, a->V, a->draft, a->draft_len, a->sampled, a->accept_len, a->next_token,
                                const_cast<int32_t*>(n.ids), n.ids_stride, const_cast<int32_t*>(n.seq_len), n.T_cap,
                                a->kv_keep_len, n.status);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const pldp_status sp = launch_sample_draws(a->logits, a->dtype, va, a->temperature, a->uniforms, a->workspace, s,
                                               "verify_sample_draft");
    if (sp != PLDP_OK) return sp;
    if (!n.H) return launch_verify_draft<NoHidden>(va, p, ixv, B, ivec, s);
    if (n.h_dtype == PLDP_BF16) return launch_verify_draft<__nv_bfloat16>(va, p, ixv, B, ivec, s);
    return launch_verify_draft<float>(va, p, ixv, B, ivec, s);
}

extern "C" PLDP_API size_t pldp_index_size(int B, int V) {
    if (B < 0 || V < 1) return 0;
    return index_layout(B, V).total;
}

extern "C" PLDP_API pldp_status pldp_index_build(const int32_t* ids, int64_t ids_stride, const int32_t* seq_len,
                                                 int B, int64_t T_cap, int V, void* index, size_t index_bytes,
                                                 uint32_t* status, void* stream) {
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "index_build: B < 0");
    if (B > 65535) return fail(PLDP_ERR_UNSUPPORTED, "index_build: B > 65535");
    if (V < 1) return fail(PLDP_ERR_INVALID_ARG, "index_build: V < 1");
    if (T_cap < 0 || T_cap > kMaxPositions) return fail(PLDP_ERR_INVALID_ARG, "index_build: T_cap outside [0, 2^27]");
    if (ids_stride < T_cap) return fail(PLDP_ERR_INVALID_ARG, "index_build: ids_stride < T_cap");
    if (B == 0) return PLDP_OK;
    if (!ids || !seq_len || !index) return fail(PLDP_ERR_INVALID_ARG, "index_build: null pointer");
    const size_t need = index_layout(B, V).total;
    if (index_bytes < need || !aligned16(index))
        return fail(PLDP_ERR_INVALID_ARG, "index_build: index needs %zu bytes, 16-byte aligned", need);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemsetAsync(index, 0, need, s);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "index_build: clearing the index: %s", cudaGetErrorString(e));
    const IndexView ix = index_view(index, B, V);
    int64_t chunks = (T_cap + 8191) / 8192;
    if (chunks < 1) chunks = 1;
    if (chunks > 65535) chunks = 65535;
    e = launch_pdl(index_build_kernel, dim3(static_cast<unsigned>(chunks), static_cast<unsigned>(B)), dim3(kThreads), 0,
                   s, 0, ids, ids_stride, seq_len, T_cap, ix);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "index_build: launch failed: %s", cudaGetErrorString(e));
    e = launch_pdl(index_finish_kernel, dim3(static_cast<unsigned>((B + 255) / 256)), dim3(256), 0, s, 0, seq_len, B,
                   T_cap, ix, status);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "index_build: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}
