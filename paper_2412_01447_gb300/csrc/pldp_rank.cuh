// Candidate ranking of PLD+ as device building blocks shared by pldp_rank_hidden,
// pldp_rank_attention and pldp_draft_step:
//   hidden states -- Eq. 3 (Sec. 4.2.2): score_j = cos(H_{j-1}, H_{t-1})
//   attentions    -- Eq. 2 (Sec. 4.2.1): score_j = max over the selected (layer, head)
//                    rows of the attention of query t-1 to key j (or their sum)
//
// S CTAs serve a sequence; candidate i belongs to CTA i mod S.  A CTA scores its
// candidates P at a time (P = 1, 2, 4 or 8, the largest not above its count)
// with 8 / P warps per candidate, each warp taking an interleaved share of the
// row, so that one candidate is read by the whole CTA in one DRAM round trip.
// Partial sums meet in shared memory and are combined in a fixed order: results
// are deterministic.  With 8 or more candidates per CTA (one warp per candidate)
// the warps run on their own instead: each streams its candidates in turn with
// no CTA barrier between them, and keeps the rows of its next candidates coming
// into L2 with bulk prefetches, so that many rows are in flight per SM.
//
// Argmax keys pack (score, position): the larger score wins, equal scores go to
// the smaller position, whatever the order of reduction.
#pragma once

#include <math.h>

#include "pldp_internal.cuh"

namespace pldp {

constexpr int kRankThreads = 256;
constexpr int kRankWarps = kRankThreads / 32;
constexpr int kRowUnroll = 8;                 // 16-byte loads in flight per lane
constexpr int kLookahead = 2;                 // candidates per warp whose rows are prefetched into L2
#ifdef PLDP_TEST_STUCK_QUERY_WAIT
constexpr uint32_t kQueryPolls = 1u << 12;    // test build: a short bound on the wait for the query row
#else
constexpr uint32_t kQueryPolls = kMbarPolls;
#endif

// Brings `bytes` (a multiple of 16, 16-byte aligned) at ptr into L2: one bulk
// prefetch, no registers held, no completion to wait for.
__device__ __forceinline__ void prefetch_l2_bulk(const void* ptr, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(ptr), "r"(bytes) : "memory");
}

struct RankShared {
    float part[kRankWarps][3];                 // per-warp partial sums of the current batch
    unsigned long long slot_key[kRankWarps];   // best key seen by each candidate slot
    int32_t jpre[kRankWarps];                  // prefetched positions of the first batch
    int err;
};

struct Batch {
    int n_local, P, G, slot, sub;
};

// A group of NW warps (first warp w0) that ranks on its own, synchronising on
// named barrier `bar` (0 = the whole CTA, i.e. __syncthreads when NW = 8).
struct WarpGroup {
    int w0, nw, bar;
    __device__ __forceinline__ int warp() const { return (static_cast<int>(threadIdx.x) >> 5) - w0; }
    __device__ __forceinline__ void sync() const {
        asm volatile("bar.sync %0, %1;" ::"r"(bar), "r"(nw * 32) : "memory");
    }
};

__device__ __forceinline__ WarpGroup whole_cta() { return WarpGroup{0, kRankWarps, 0}; }

__device__ __forceinline__ Batch batch_shape(int n, int S, int rank, const WarpGroup& wg) {
    const int warp = wg.warp();
    const int pmax = wg.nw;   // 8 or 4
    Batch bt;
    bt.n_local = (n > rank) ? (n - rank + S - 1) / S : 0;
    bt.P = (bt.n_local >= 8 && pmax >= 8) ? 8 : (bt.n_local >= 4 ? 4 : (bt.n_local >= 2 ? 2 : 1));
    if (bt.P > pmax) bt.P = pmax;
    bt.G = wg.nw / bt.P;
    bt.slot = warp / bt.G;
    bt.sub = warp - bt.slot * bt.G;
    return bt;
}

__device__ __forceinline__ void rank_shared_init(RankShared& sh) {
    if (threadIdx.x < kRankWarps) sh.slot_key[threadIdx.x] = 0;
    if (threadIdx.x == 0) sh.err = 0;
}

__device__ __forceinline__ unsigned long long rank_best_key(const RankShared& sh) {
    unsigned long long k = 0;
#pragma unroll
    for (int w = 0; w < kRankWarps; ++w) k = sh.slot_key[w] > k ? sh.slot_key[w] : k;
    return k;
}

template <typename T>
__device__ __forceinline__ void accum16(const uint4& a, const uint4& q, float& dot, float& na,
                                        float& nq);

template <>
__device__ __forceinline__ void accum16<__nv_bfloat16>(const uint4& a, const uint4& q, float& dot,
                                                       float& na, float& nq) {
    const uint32_t av[4] = {a.x, a.y, a.z, a.w};
    const uint32_t qv[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float a0 = __uint_as_float(av[k] << 16), a1 = __uint_as_float(av[k] & 0xFFFF0000u);
        const float q0 = __uint_as_float(qv[k] << 16), q1 = __uint_as_float(qv[k] & 0xFFFF0000u);
        dot = fmaf(a0, q0, dot);
        dot = fmaf(a1, q1, dot);
        na = fmaf(a0, a0, na);
        na = fmaf(a1, a1, na);
        nq = fmaf(q0, q0, nq);
        nq = fmaf(q1, q1, nq);
    }
}

template <>
__device__ __forceinline__ void accum16<float>(const uint4& a, const uint4& q, float& dot,
                                               float& na, float& nq) {
    const uint32_t av[4] = {a.x, a.y, a.z, a.w};
    const uint32_t qv[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float x = __uint_as_float(av[k]), y = __uint_as_float(qv[k]);
        dot = fmaf(x, y, dot);
        na = fmaf(x, x, na);
        nq = fmaf(y, y, nq);
    }
}

// cos = dot / sqrt(|a|^2 |q|^2); a zero norm gives 0 (the library's stated reading).
// fp32 throughout (the double-precision units of this GPU are few); the two
// reciprocal square roots keep the product of the norms from overflowing.
__device__ __forceinline__ float finish_cosine(float dot, float na, float nq) {
    if (na == 0.0f || nq == 0.0f) return 0.0f;
    return dot * rsqrtf(na) * rsqrtf(nq);
}

// Position of this CTA's k-th candidate (list index i): the first batch's from
// `jpre` (shared), the others from the candidate row.
template <bool CANDS_SHARED>
__device__ __forceinline__ int64_t cand_at(const int32_t* __restrict__ cands, const int32_t* jpre, int k, int i,
                                           int P) {
    if (k < P && jpre) return jpre[k];
    return CANDS_SHARED ? cands[i] : __ldcg(cands + i);
}

// Eq. 3 with one warp per candidate (G = 1): warp `slot` scores candidates slot,
// slot + P, ... of this CTA on its own.  Lane 0 keeps the rows of the warp's next
// kLookahead candidates on their way into L2; their positions are read one
// iteration before they are needed, so the prefetches never wait.
template <typename T, bool CANDS_SHARED>
__device__ __forceinline__ void hidden_rank_warp(const T* __restrict__ hb, int64_t d, int64_t t,
                                                 const int32_t* __restrict__ cands, int S, int rank,
                                                 const int32_t* jpre, const T* q_sh, uint64_t* bar, bool q_pending,
                                                 float threshold, float* __restrict__ scores_row, RankShared& sh,
                                                 const Batch& bt) {
    constexpr int E = 16 / sizeof(T);
    const int lane = threadIdx.x & 31;
    const int P = bt.P;
    const int64_t nch = d / E;
    const uint32_t row_bytes = static_cast<uint32_t>(d * sizeof(T));
    auto cand = [&](int k) -> int64_t { return cand_at<CANDS_SHARED>(cands, jpre, k, rank + S * k, P); };
    auto prefetch_row = [&](int64_t j) {
        if (j >= 1 && j < t) prefetch_l2_bulk(hb + (j - 1) * d, row_bytes);
    };
    int64_t jnext = -1;                                   // lane 0: position of candidate k + kLookahead * P
    if (lane == 0) {
        for (int a = 1; a < kLookahead; ++a)
            if (bt.slot + a * P < bt.n_local) prefetch_row(cand(bt.slot + a * P));
        if (bt.slot + kLookahead * P < bt.n_local) jnext = cand(bt.slot + kLookahead * P);
    }
    bool q_ready = !q_pending, timed_out = false;
    unsigned long long best = 0;
    for (int k = bt.slot; k < bt.n_local; k += P) {
        const int i = rank + S * k;
        const int64_t j = cand(k);
        if (lane == 0) {
            prefetch_row(jnext);
            const int kn = k + (kLookahead + 1) * P;
            jnext = kn < bt.n_local ? cand(kn) : -1;
        }
        const bool ok = j >= 1 && j < t;
        float dot = 0.f, na = 0.f, nq = 0.f;
        if (ok) {
            const T* row = hb + (j - 1) * d;              // H_{j-1}
            for (int64_t c0 = lane; c0 < nch; c0 += 32 * kRowUnroll) {
                uint4 a[kRowUnroll];
#pragma unroll
                for (int u = 0; u < kRowUnroll; ++u) {
                    const int64_t c = c0 + 32 * u;
                    if (c < nch) a[u] = ld_stream16(row + c * E);
                }
                if (!q_ready) {
                    if (!mbar_wait(bar, 0, kQueryPolls)) timed_out = true;
                    q_ready = true;
                }
                if (timed_out) break;
#pragma unroll
                for (int u = 0; u < kRowUnroll; ++u) {
                    const int64_t c = c0 + 32 * u;
                    if (c < nch) {
                        const uint4 q = *reinterpret_cast<const uint4*>(q_sh + c * E);
                        accum16<T>(a[u], q, dot, na, nq);
                    }
                }
            }
        }
        if (__any_sync(0xFFFFFFFFu, timed_out)) {
            if (lane == 0) sh.err = 1;
            break;
        }
        dot = warp_sum(dot);
        na = warp_sum(na);
        nq = warp_sum(nq);
        if (lane == 0) {
            const float s = ok ? finish_cosine(0.f + dot, 0.f + na, 0.f + nq) : -INFINITY;   // as the CTA path sums
            if (scores_row) scores_row[i] = s;
            if (ok && s > threshold) {
                const unsigned long long key = pack_key(s, static_cast<uint32_t>(j));
                best = key > best ? key : best;
            }
        }
    }
    if (lane == 0 && best > sh.slot_key[bt.slot]) sh.slot_key[bt.slot] = best;
}

// Eq. 3 for this CTA's candidates.  `hb` is the sequence's hidden slice, `cands`
// its candidate row, `q_sh` the query row H_{t-1} in shared memory -- complete,
// or (q_pending) still arriving through `bar`, waited for before its first use.
// Scores go to scores_row[i] (if given); keys of eligible candidates to
// sh.slot_key.  CTA-uniform call; `jpre` (optional, shared) holds the first
// batch's positions.  Returns with sh.err set if the query never arrived.
// With CANDS_SHARED the candidate list is in shared memory (else global, read
// through L2 since other CTAs of the cluster may have just written it).
template <typename T, bool VEC, bool CANDS_SHARED = false>
__device__ __forceinline__ void hidden_rank_cta(const T* __restrict__ hb, int64_t d, int64_t t,
                                                const int32_t* __restrict__ cands, int n, int S,
                                                int rank, const int32_t* jpre, const T* q_sh,
                                                uint64_t* bar, bool q_pending, float threshold,
                                                float* __restrict__ scores_row, RankShared& sh,
                                                const WarpGroup& wg = whole_cta()) {
    const int lane = threadIdx.x & 31, warp = wg.warp();
    const Batch bt = batch_shape(n, S, rank, wg);
    if constexpr (VEC) {
        if (bt.G == 1) {                                  // one warp per candidate: no barriers
            hidden_rank_warp<T, CANDS_SHARED>(hb, d, t, cands, S, rank, jpre, q_sh, bar, q_pending, threshold,
                                              scores_row, sh, bt);
            wg.sync();
            return;
        }
    }
    bool q_ready = !q_pending, timed_out = false;
    for (int k0 = 0; k0 < bt.n_local; k0 += bt.P) {
        const int k = k0 + bt.slot;
        const bool active = k < bt.n_local;
        const int i = rank + S * k;
        int64_t j = -1;
        if (active) j = (k0 == 0 && jpre) ? jpre[k] : (CANDS_SHARED ? cands[i] : __ldcg(cands + i));
        const bool ok = active && j >= 1 && j < t;
        float dot = 0.f, na = 0.f, nq = 0.f;
        if (ok) {
            const T* row = hb + (j - 1) * d;              // H_{j-1}
            if constexpr (VEC) {
                constexpr int E = 16 / sizeof(T);
                const int64_t nch = d / E;
                const int64_t step = static_cast<int64_t>(bt.G) * 32;
                for (int64_t c0 = bt.sub * 32 + lane; c0 < nch; c0 += step * kRowUnroll) {
                    uint4 a[kRowUnroll];
#pragma unroll
                    for (int u = 0; u < kRowUnroll; ++u) {
                        const int64_t c = c0 + step * u;
                        if (c < nch) a[u] = ld_stream16(row + c * E);
                    }
                    if (!q_ready) {
                        if (!mbar_wait(bar, 0, kQueryPolls)) timed_out = true;
                        q_ready = true;
                    }
                    if (timed_out) break;
#pragma unroll
                    for (int u = 0; u < kRowUnroll; ++u) {
                        const int64_t c = c0 + step * u;
                        if (c < nch) {
                            const uint4 q = *reinterpret_cast<const uint4*>(q_sh + c * E);
                            accum16<T>(a[u], q, dot, na, nq);
                        }
                    }
                }
            } else {
                for (int64_t c = bt.sub * 32 + lane; c < d; c += static_cast<int64_t>(bt.G) * 32) {
                    const float x = to_f32(row[c]), y = to_f32(q_sh[c]);
                    dot = fmaf(x, y, dot);
                    na = fmaf(x, x, na);
                    nq = fmaf(y, y, nq);
                }
            }
        }
        dot = warp_sum(dot);
        na = warp_sum(na);
        nq = warp_sum(nq);
        if (lane == 0) {
            sh.part[warp][0] = dot;
            sh.part[warp][1] = na;
            sh.part[warp][2] = nq;
        }
        if (__any_sync(0xFFFFFFFFu, timed_out) && lane == 0) sh.err = 1;
        wg.sync();
        if (bt.sub == 0 && lane == 0 && active) {
            float s = -INFINITY;
            if (ok) {
                float D = 0.f, A = 0.f, Q = 0.f;
                for (int g = 0; g < bt.G; ++g) {          // fixed order
                    D += sh.part[warp + g][0];
                    A += sh.part[warp + g][1];
                    Q += sh.part[warp + g][2];
                }
                s = finish_cosine(D, A, Q);
            }
            if (scores_row) scores_row[i] = s;
            if (ok && s > threshold) {
                const unsigned long long key = pack_key(s, static_cast<uint32_t>(j));
                if (key > sh.slot_key[bt.slot]) sh.slot_key[bt.slot] = key;
            }
        }
        wg.sync();
        if (sh.err) break;                                // group-uniform after the barrier
    }
}

// One attention value, dtype chosen at run time (bf16 when a_bf16).
__device__ __forceinline__ float load_attn(const void* base, int64_t idx, bool a_bf16) {
    if (a_bf16) return __bfloat162float(static_cast<const __nv_bfloat16*>(base)[idx]);
    return static_cast<const float*>(base)[idx];
}

// Eq. 2 with one warp per candidate (G = 1): warp `slot` takes candidates slot,
// slot + P, ... of this CTA two at a time, on its own (no CTA barrier), so twice
// the scattered values are in flight.  Lane sums run in the order of the CTA path.
template <bool CANDS_SHARED>
__device__ __forceinline__ void attention_rank_warp(const void* ab, bool a_bf16, const int64_t* rows_sh, int n_sel,
                                                    int64_t key_stride, int64_t t, const int32_t* __restrict__ cands,
                                                    int S, int rank,
                                                    const int32_t* jpre, bool is_max, float* __restrict__ scores_row,
                                                    RankShared& sh, const Batch& bt) {
    const int lane = threadIdx.x & 31;
    const int P = bt.P;
    constexpr int U = 4;
    unsigned long long best = 0;
    for (int k = bt.slot; k < bt.n_local; k += 2 * P) {
        int64_t j[2];
        bool act[2], ok[2];
        float acc[2];
#pragma unroll
        for (int c = 0; c < 2; ++c) {
            const int kk = k + c * P;
            act[c] = kk < bt.n_local;
            j[c] = act[c] ? cand_at<CANDS_SHARED>(cands, jpre, kk, rank + S * kk, P) : -1;
            ok[c] = act[c] && j[c] >= 0 && j[c] < t;
            acc[c] = is_max ? -INFINITY : 0.0f;
        }
        for (int r0 = lane; r0 < n_sel; r0 += 32 * U) {
            float v[2][U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int r = r0 + 32 * u;
                const int64_t off = (r < n_sel) ? rows_sh[r] : -1;
#pragma unroll
                for (int c = 0; c < 2; ++c)
                    v[c][u] = (ok[c] && off >= 0) ? load_attn(ab, off + j[c] * key_stride, a_bf16) : NAN;
            }
#pragma unroll
            for (int c = 0; c < 2; ++c)
#pragma unroll
                for (int u = 0; u < U; ++u)
                    if (v[c][u] == v[c][u]) acc[c] = is_max ? fmaxf(acc[c], v[c][u]) : acc[c] + v[c][u];
        }
#pragma unroll
        for (int c = 0; c < 2; ++c) {
            if (is_max) {
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) acc[c] = fmaxf(acc[c], __shfl_xor_sync(0xFFFFFFFFu, acc[c], o));
            } else {
                acc[c] = warp_sum(acc[c]);
            }
        }
        if (lane == 0) {
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                if (!act[c]) continue;
                const float s = ok[c] ? acc[c] : -INFINITY;
                if (scores_row) scores_row[rank + S * (k + c * P)] = s;
                if (ok[c]) {
                    const unsigned long long key = pack_key(s, static_cast<uint32_t>(j[c]));
                    best = key > best ? key : best;
                }
            }
        }
    }
    if (lane == 0 && best > sh.slot_key[bt.slot]) sh.slot_key[bt.slot] = best;
}

// Eq. 2 under MAX with one warp per candidate when the selected rows of a key are
// one dense run of nv 16-byte vectors (all R rows in order, row stride 1: the
// key-major layout; nv a power of two, at most 32 * kDenseLoads): the warp reads
// whole vectors -- up to kDenseLoads per lane in flight, 32 * kDenseLoads vectors,
// i.e. several candidates' runs at once when they are short -- instead of one value
// per lane.  A lane's vectors belong to one candidate per load; the max over the
// nv lanes (nv <= 32) or the nv / 32 loads and the warp (nv > 32) of a candidate is
// exact, so the scores are those of the value-per-lane path bit for bit.
constexpr int kDenseLoads = 4;

template <typename T, bool CANDS_SHARED>
__device__ __forceinline__ void attention_rank_warp_dense(const T* ab, int nv, int64_t key_stride, int64_t t,
                                                          const int32_t* __restrict__ cands, int S, int rank,
                                                          const int32_t* jpre, float* __restrict__ scores_row,
                                                          RankShared& sh, const Batch& bt) {
    constexpr int VW = 16 / static_cast<int>(sizeof(T));
    const int lane = threadIdx.x & 31;
    const int P = bt.P;
    const int lpc = nv < 32 ? nv : 32;                    // lanes per candidate and load
    const int cpl = 32 / lpc;                             // candidates per load
    const int vpl = nv / lpc;                             // loads per lane per candidate (<= kDenseLoads)
    const int ng = kDenseLoads / vpl;                     // load groups (one candidate per lane each)
    unsigned long long best = 0;
    for (int i0 = 0; bt.slot + i0 * P < bt.n_local; i0 += ng * cpl) {   // warp-uniform
        uint4 x[kDenseLoads];
        int32_t jl[kDenseLoads];                          // this lane's candidate position in load u, or -1
#pragma unroll
        for (int u = 0; u < kDenseLoads; ++u) {
            const int g = u / vpl;                        // the load group (vpl: 1, 2 or 4)
            const int k = bt.slot + (i0 + g * cpl + lane / lpc) * P;
            int32_t j = -1;
            if (k < bt.n_local) {
                const int64_t jj = cand_at<CANDS_SHARED>(cands, jpre, k, rank + S * k, P);
                if (jj >= 0 && jj < t) j = static_cast<int32_t>(jj);
            }
            jl[u] = j;
            if (j >= 0)
                x[u] = *reinterpret_cast<const uint4*>(
                    ab + j * key_stride + static_cast<int64_t>((u - g * vpl) * lpc + lane % lpc) * VW);
        }
        float m[kDenseLoads];
#pragma unroll
        for (int u = 0; u < kDenseLoads; ++u) m[u] = jl[u] >= 0 ? vmax(x[u], T()) : -INFINITY;
        // fold each group's vpl loads into its first (registers only: the indices are fixed)
#pragma unroll
        for (int st = 1; st < kDenseLoads; st <<= 1)
#pragma unroll
            for (int u = 0; u + st < kDenseLoads; u += 2 * st)
                if (st < vpl) m[u] = fmaxf(m[u], m[u + st]);
        // then over the candidate's lanes; lane q * lpc writes candidate i0 + g * cpl + q
#pragma unroll
        for (int u = 0; u < kDenseLoads; ++u) {
            if (u % vpl != 0) continue;                   // warp-uniform
            float v = m[u];
            for (int o = lpc / 2; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
            const int k = bt.slot + (i0 + (u / vpl) * cpl + lane / lpc) * P;
            if (lane % lpc == 0 && k < bt.n_local) {
                const int32_t j = jl[u];
                const float sc = j >= 0 ? v : -INFINITY;
                if (scores_row) scores_row[rank + S * k] = sc;
                if (j >= 0) {
                    const unsigned long long key = pack_key(sc, static_cast<uint32_t>(j));
                    best = key > best ? key : best;
                }
            }
        }
    }
    best = warp_max_u64(best);
    if (lane == 0 && best > sh.slot_key[bt.slot]) sh.slot_key[bt.slot] = best;
}

// Eq. 2 for this CTA's candidates.  `rows_sh` (shared) holds the element offset
// of each selected row, or -1 for an invalid one; key j of a row is key_stride
// elements after key j - 1.  Same conventions as
// hidden_rank_cta; every candidate in [0, t) is eligible.  With CANDS_SHARED
// the candidate list is in shared memory (else global, read through L2).
template <bool CANDS_SHARED = false>
__device__ __forceinline__ void attention_rank_cta(const void* ab, bool a_bf16,
                                                   const int64_t* rows_sh, int n_sel, int64_t key_stride, int64_t t,
                                                   const int32_t* __restrict__ cands, int n, int S,
                                                   int rank, const int32_t* jpre, bool is_max,
                                                   float* __restrict__ scores_row, RankShared& sh,
                                                   const WarpGroup& wg = whole_cta(), int dense_nv = 0) {
    const int lane = threadIdx.x & 31, warp = wg.warp();
    const Batch bt = batch_shape(n, S, rank, wg);
    if (bt.G == 1 && dense_nv > 0 && is_max) {            // one warp per candidate, whole vectors
        if (a_bf16)
            attention_rank_warp_dense<__nv_bfloat16, CANDS_SHARED>(static_cast<const __nv_bfloat16*>(ab), dense_nv,
                                                                   key_stride, t, cands, S, rank, jpre, scores_row,
                                                                   sh, bt);
        else
            attention_rank_warp_dense<float, CANDS_SHARED>(static_cast<const float*>(ab), dense_nv, key_stride, t,
                                                           cands, S, rank, jpre, scores_row, sh, bt);
        wg.sync();
        return;
    }
    if (bt.G == 1) {                                      // one warp per candidate: no barriers
        attention_rank_warp<CANDS_SHARED>(ab, a_bf16, rows_sh, n_sel, key_stride, t, cands, S, rank, jpre, is_max,
                                          scores_row, sh, bt);
        wg.sync();
        return;
    }
    constexpr int U = 4;
    for (int k0 = 0; k0 < bt.n_local; k0 += bt.P) {
        const int k = k0 + bt.slot;
        const bool active = k < bt.n_local;
        const int i = rank + S * k;
        int64_t j = -1;
        if (active) j = (k0 == 0 && jpre) ? jpre[k] : (CANDS_SHARED ? cands[i] : __ldcg(cands + i));
        const bool ok = active && j >= 0 && j < t;
        float acc = is_max ? -INFINITY : 0.0f;
        if (ok) {
            const int step = bt.G * 32;
            for (int r0 = bt.sub * 32 + lane; r0 < n_sel; r0 += step * U) {
                float v[U];
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int r = r0 + step * u;
                    const int64_t off = (r < n_sel) ? rows_sh[r] : -1;
                    v[u] = (off >= 0) ? load_attn(ab, off + j * key_stride, a_bf16) : NAN;
                }
#pragma unroll
                for (int u = 0; u < U; ++u)
                    if (v[u] == v[u]) acc = is_max ? fmaxf(acc, v[u]) : acc + v[u];
            }
        }
        if (is_max) {
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) acc = fmaxf(acc, __shfl_xor_sync(0xFFFFFFFFu, acc, o));
        } else {
            acc = warp_sum(acc);
        }
        if (lane == 0) sh.part[warp][0] = acc;
        wg.sync();
        if (bt.sub == 0 && lane == 0 && active) {
            float s = -INFINITY;
            if (ok) {
                s = sh.part[warp][0];
                for (int g = 1; g < bt.G; ++g)          // fixed order
                    s = is_max ? fmaxf(s, sh.part[warp + g][0]) : s + sh.part[warp + g][0];
            }
            if (scores_row) scores_row[i] = s;
            if (ok) {
                const unsigned long long key = pack_key(s, static_cast<uint32_t>(j));
                if (key > sh.slot_key[bt.slot]) sh.slot_key[bt.slot] = key;
            }
        }
        wg.sync();
    }
}

// Host: the attention layout rules of the ranking calls (A + b*seq_stride +
// r*row_stride + key*key_stride, rows that do not overlap).  Returns null when the
// layout is valid, else what is wrong.
inline const char* attention_layout_error(int R, int64_t T_cap, int64_t row_stride, int64_t key_stride,
                                          int64_t seq_stride) {
    if (row_stride < 1 || key_stride < 1) return "row and key strides must be >= 1";
    const bool head_major = row_stride >= T_cap * key_stride;
    const bool key_major = key_stride >= static_cast<int64_t>(R) * row_stride;
    if (!head_major && !key_major) return "rows overlap: need row_stride >= T_cap*key_stride or key_stride >= R*row_stride";
    const int64_t extent = static_cast<int64_t>(R - 1) * row_stride + (T_cap > 0 ? T_cap - 1 : 0) * key_stride + 1;
    if (seq_stride < extent) return "seq_stride shorter than one sequence's rows";
    return nullptr;
}

// Stages the element offsets of the selected attention rows; returns (in every
// thread, after a barrier) whether some row index was outside [0, R).
__device__ __forceinline__ bool stage_rows(int64_t* rows_sh, const int32_t* row_idx, int n_sel, int R,
                                           int64_t row_stride, int* bad_flag) {
    if (threadIdx.x == 0) *bad_flag = 0;
    __syncthreads();
    for (int k = threadIdx.x; k < n_sel; k += kRankThreads) {
        const int r = row_idx ? row_idx[k] : k;
        const bool okr = (r >= 0 && r < R);
        rows_sh[k] = okr ? static_cast<int64_t>(r) * row_stride : -1;
        if (!okr) *bad_flag = 1;
    }
    __syncthreads();
    return *bad_flag != 0;
}

}  // namespace pldp
