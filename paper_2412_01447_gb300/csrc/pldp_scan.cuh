// Candidate scan of PLD+ -- Eq. 1 (Sec. 4.2) with the longest-suffix n-gram rule --
// as device building blocks shared by pldp_find_candidates and pldp_draft_step.
//
// The S CTAs of a cluster each own a contiguous chunk of one sequence.  Pass 1
// streams the chunk (16-byte loads when rows are aligned) and counts, for every
// n, the positions whose suffix match with x_t reaches n.  The counts are read
// across the cluster over distributed shared memory; n* is the longest n with a
// match anywhere, and a CTA's matches go after those of lower-ranked CTAs.
// Pass 2 (only in CTAs that own matches of length n*) rescans the chunk and
// writes the positions in ascending order with warp scans.
#pragma once

#include "pldp_internal.cuh"

namespace pldp {

constexpr int kScanThreads = 256;
constexpr int kScanWarps = kScanThreads / 32;
constexpr int kScanUnroll = 8;          // 16-byte loads in flight per thread in pass 1
constexpr int kScanMaxCluster = 8;      // portable cluster size

struct ScanShared {
    int cnt[PLDP_MAX_NGRAM + 1];                   // cnt[n]: positions with match length >= n
    int table[kScanMaxCluster][PLDP_MAX_NGRAM + 1];
    int warp_tot[kScanWarps];
    int nstar, offset, mine, total;
};

// How ids are read: through the read-only cache (a context that no kernel of
// the call writes), or through L2 (a context that the same kernel has just
// appended to, which the read-only path is not guaranteed to see).
struct ReadOnlyIds {
    static __device__ __forceinline__ int32_t one(const int32_t* p) { return __ldg(p); }
    static __device__ __forceinline__ int4 four(const int4* p) { return __ldg(p); }
};
struct CoherentIds {
    static __device__ __forceinline__ int32_t one(const int32_t* p) { return __ldcg(p); }
    static __device__ __forceinline__ int4 four(const int4* p) { return __ldcg(p); }
};

// Length of the common suffix of x[0..j] and x[0..t] (x_j == x_t already known),
// capped at n_max.  j < t, so x_{t-m} exists whenever x_{j-m} does.  Every
// thread of the CTA reads the same few suffix tokens.
template <typename RD = ReadOnlyIds>
__device__ __forceinline__ int suffix_match(const int32_t* __restrict__ row, int64_t j, int64_t t,
                                            int n_max) {
    int m = 1;
    while (m < n_max && j - m >= 0 && RD::one(row + j - m) == RD::one(row + t - m)) ++m;
    return m;
}

__device__ __forceinline__ void count_hit(int (&c)[PLDP_MAX_NGRAM], int m) {
#pragma unroll
    for (int k = 0; k < PLDP_MAX_NGRAM; ++k) c[k] += (k < m) ? 1 : 0;
}

// Where pass 1 and pass 2 read the ids from: global memory (16-byte or 4-byte
// loads) or a copy of the CTA's chunk staged in shared memory (`base` = ids of
// positions c0, c0 + 1, ...).  `load4(q)` returns positions 4q .. 4q + 3.
template <typename RD>
struct GlobalIdsT {
    const int32_t* row;
    __device__ __forceinline__ int4 load4(int64_t q) const {
        return RD::four(reinterpret_cast<const int4*>(row) + q);
    }
};
using GlobalIds = GlobalIdsT<ReadOnlyIds>;
struct SharedIds {
    const int32_t* base;   // shared memory, 16-byte aligned
    int64_t q0;            // first int4 index of the staged chunk (c0 / 4)
    __device__ __forceinline__ int4 load4(int64_t q) const {
        return reinterpret_cast<const int4*>(base)[q - q0];
    }
};

// Pass 1 over positions [c0, c1) (c0 a multiple of 4 when VEC; all < t):
// c[k] += number of positions whose match length exceeds k.  With VEC the ids
// come through `src` (16-byte units); otherwise 4-byte global loads from `row`.
template <bool VEC, typename Src, typename RD = ReadOnlyIds>
__device__ __forceinline__ void scan_count(const Src& src, const int32_t* __restrict__ row, int64_t c0,
                                           int64_t c1, int64_t t, int n_max, int (&c)[PLDP_MAX_NGRAM]) {
    if (c0 >= c1) return;
    const int tid = threadIdx.x;
    const int32_t xt = RD::one(row + t);
    if constexpr (VEC) {
        const int64_t q0 = c0 >> 2, q1 = (c1 + 3) >> 2;
        for (int64_t qb = q0 + tid; qb < q1; qb += static_cast<int64_t>(kScanThreads) * kScanUnroll) {
            int4 v[kScanUnroll];
#pragma unroll
            for (int u = 0; u < kScanUnroll; ++u) {
                const int64_t q = qb + static_cast<int64_t>(u) * kScanThreads;
                if (q < q1) v[u] = src.load4(q);
            }
#pragma unroll
            for (int u = 0; u < kScanUnroll; ++u) {
                const int64_t q = qb + static_cast<int64_t>(u) * kScanThreads;
                if (q >= q1) continue;
                const int32_t e[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const int64_t p = 4 * q + k;
                    if (e[k] == xt && p < c1) count_hit(c, suffix_match<RD>(row, p, t, n_max));
                }
            }
        }
    } else {
        for (int64_t pb = c0 + tid; pb < c1; pb += static_cast<int64_t>(kScanThreads) * kScanUnroll) {
            int32_t v[kScanUnroll];
#pragma unroll
            for (int u = 0; u < kScanUnroll; ++u) {
                const int64_t p = pb + static_cast<int64_t>(u) * kScanThreads;
                if (p < c1) v[u] = RD::one(row + p);
            }
#pragma unroll
            for (int u = 0; u < kScanUnroll; ++u) {
                const int64_t p = pb + static_cast<int64_t>(u) * kScanThreads;
                if (p < c1 && v[u] == xt) count_hit(c, suffix_match<RD>(row, p, t, n_max));
            }
        }
    }
}

// Adds the per-thread counts into sh.cnt[1..n_max] (zeroed and synchronised before).
__device__ __forceinline__ void scan_reduce_counts(const int (&c)[PLDP_MAX_NGRAM], int n_max,
                                                   ScanShared& sh) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int k = 0; k < PLDP_MAX_NGRAM; ++k) {
        if (k < n_max) {
            const int s = __reduce_add_sync(0xFFFFFFFFu, c[k]);
            if (lane == 0 && s) atomicAdd(&sh.cnt[k + 1], s);
        }
    }
}

// After a cluster barrier that made every CTA's sh.cnt final: copies all CTAs'
// counts into sh.table and, in thread 0, decides n*, the total, this CTA's count
// and its output offset.  Ends with __syncthreads; issues no cluster barrier.
__device__ __forceinline__ void scan_decide(cg::cluster_group& cluster, ScanShared& sh, int CL,
                                            int rank, int ngram_min, int ngram_max) {
    const int tid = threadIdx.x;
    for (int i = tid; i < CL * (PLDP_MAX_NGRAM + 1); i += kScanThreads) {
        const int r = i / (PLDP_MAX_NGRAM + 1), n = i % (PLDP_MAX_NGRAM + 1);
        const int* remote = cluster.map_shared_rank(&sh.cnt[0], r);
        sh.table[r][n] = remote[n];
    }
    __syncthreads();
    if (tid == 0) {
        int nstar = 0, total = 0;
        for (int n = ngram_max; n >= ngram_min; --n) {
            int tot = 0;
            for (int r = 0; r < CL; ++r) tot += sh.table[r][n];
            if (tot > 0) {
                nstar = n;
                total = tot;
                break;
            }
        }
        int off = 0;
        if (nstar)
            for (int r = 0; r < rank; ++r) off += sh.table[r][nstar];
        sh.nstar = nstar;
        sh.total = total;
        sh.offset = off;
        sh.mine = nstar ? sh.table[rank][nstar] : 0;
    }
    __syncthreads();
}

// Pass 2: writes this CTA's matches of length >= nstar, in ascending order, to
// dst[sh.offset ...] (entries at or past C_cap are dropped).  CTA-uniform call.
// `on_write(j)` is called by the thread that writes position j.
struct NoHook {
    __device__ __forceinline__ void operator()(int64_t) const {}
};

template <bool VEC, typename Src, typename Hook = NoHook, typename RD = ReadOnlyIds>
__device__ __forceinline__ void scan_write(const Src& src, const int32_t* __restrict__ row, int64_t c0,
                                           int64_t c1, int64_t t, int n_max, ScanShared& sh,
                                           int32_t* __restrict__ dst, int C_cap,
                                           const Hook& on_write = Hook()) {
    const int nstar = sh.nstar, mine = sh.mine;
    int64_t out = sh.offset;
    if (!(nstar > 0 && mine > 0 && out < C_cap)) return;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int32_t xt = RD::one(row + t);
    const int64_t end = out + mine;
    constexpr int G = VEC ? 4 : 1;                       // positions per thread per tile
    const int64_t g0 = c0 / G, g1 = (c1 + G - 1) / G;
    for (int64_t gb = g0; gb < g1 && out < end && out < C_cap; gb += kScanThreads) {
        const int64_t g = gb + tid;
        uint32_t mask = 0;
        if (g < g1) {
            int32_t e[G];
            if constexpr (VEC) {
                const int4 v = src.load4(g);
                e[0] = v.x;
                e[1] = v.y;
                e[2] = v.z;
                e[3] = v.w;
            } else {
                e[0] = RD::one(row + g);
            }
#pragma unroll
            for (int k = 0; k < G; ++k) {
                const int64_t p = g * G + k;
                if (e[k] == xt && p < c1 && suffix_match<RD>(row, p, t, n_max) >= nstar) mask |= 1u << k;
            }
        }
        const int cnt = __popc(mask);
        int incl = cnt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o) incl += v;
        }
        if (lane == 31) sh.warp_tot[warp] = incl;
        __syncthreads();
        int before = 0, tile = 0;
#pragma unroll
        for (int w = 0; w < kScanWarps; ++w) {
            const int x = sh.warp_tot[w];
            before += (w < warp) ? x : 0;
            tile += x;
        }
        int64_t pos = out + before + (incl - cnt);
        while (mask) {
            const int k = __ffs(mask) - 1;
            mask &= mask - 1;
            if (pos < C_cap) {
                dst[pos] = static_cast<int32_t>(g * G + k);
                on_write(g * G + k);
            }
            ++pos;
        }
        out += tile;
        __syncthreads();   // warp_tot is rewritten by the next tile
    }
}

__device__ __forceinline__ void cluster_arrive() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Cluster size and chunk for scanning T_cap positions of B sequences: one CTA per
// `per_cta` positions, at most a portable cluster, and no more CTAs in all than
// `resident` (so the grid is a single wave).
inline void scan_shape(int64_t T_cap, int B, int resident, int64_t per_cta, int* CL_out,
                       int64_t* chunk_out) {
    int CL = static_cast<int>((T_cap + per_cta - 1) / per_cta);
    const int per_seq = resident / (B > 0 ? B : 1);
    if (CL > per_seq) CL = per_seq;
    CL = CL < 1 ? 1 : (CL > kScanMaxCluster ? kScanMaxCluster : CL);
    int64_t chunk = (T_cap + CL - 1) / CL;
    chunk = (chunk + 3) / 4 * 4;
    if (chunk < 4) chunk = 4;
    *CL_out = CL;
    *chunk_out = chunk;
}

}  // namespace pldp
