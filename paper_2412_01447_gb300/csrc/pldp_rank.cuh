// Candidate ranking of PLD+ as device building blocks shared by pldp_rank_hidden,
// pldp_rank_attention and pldp_draft_step:
//   hidden states -- Eq. 3 (Sec. 4.2.2): score_j = cos(H_{j-1}, H_{t-1})
//   attentions    -- Eq. 2 (Sec. 4.2.1): score_j = max over the selected (layer, head)
//                    rows of the attention of query t-1 to key j (or their sum)
//
// S CTAs serve a sequence; candidate i belongs to CTA i mod S.  A CTA scores its
// candidates P at a time (P = 1, 2, 4 or 8, the largest not above its count)
// with 8 / P warps per candidate, each warp taking an interleaved share of the
// row, so that one candidate is read by the whole CTA in one DRAM round trip
// while many candidates stream with one warp each.  Partial sums meet in shared
// memory and are combined in a fixed order: results are deterministic.
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
                        if (!mbar_wait(bar, 0, kMbarPolls)) timed_out = true;
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

// Eq. 2 for this CTA's candidates.  `rows_sh` (shared) holds the element offset
// of each selected row, or -1 for an invalid one.  Same conventions as
// hidden_rank_cta; every candidate in [0, t) is eligible.  With CANDS_SHARED
// the candidate list is in shared memory (else global, read through L2).
template <bool CANDS_SHARED = false>
__device__ __forceinline__ void attention_rank_cta(const void* ab, bool a_bf16,
                                                   const int64_t* rows_sh, int n_sel, int64_t t,
                                                   const int32_t* __restrict__ cands, int n, int S,
                                                   int rank, const int32_t* jpre, bool is_max,
                                                   float* __restrict__ scores_row, RankShared& sh,
                                                   const WarpGroup& wg = whole_cta()) {
    const int lane = threadIdx.x & 31, warp = wg.warp();
    const Batch bt = batch_shape(n, S, rank, wg);
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
                    v[u] = (off >= 0) ? load_attn(ab, off + j, a_bf16) : NAN;
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
