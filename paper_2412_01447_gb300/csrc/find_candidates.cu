// Candidate search of PLD+ -- Eq. 1 (Sec. 4.2) with the longest-suffix n-gram rule.
//
// One thread-block cluster per sequence.  Each CTA of the cluster scans a
// contiguous chunk of the context with 16-byte loads (pass 1), counting, for
// every n-gram length n, the positions whose suffix match reaches n.  The
// counts are exchanged through distributed shared memory: every CTA learns the
// chosen n* (the longest length with a match anywhere) and how many matches the
// lower-ranked CTAs own, which is where its own matches go in the ascending
// list.  Only CTAs that own matches of length n* rescan their chunk (pass 2) to
// write them, compacting in order with warp scans.  Matches are rare on real
// contexts, so the common cost is one streaming read of the ids.
#include "pldp_internal.cuh"

namespace pldp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 8;          // 16-byte loads in flight per thread in pass 1
constexpr int kMaxCluster = 8;      // portable cluster size
constexpr int64_t kPositionsPerCta = 4096;

struct FindShared {
    int cnt[PLDP_MAX_NGRAM + 1];                   // cnt[n]: positions with match length >= n
    int32_t suffix[PLDP_MAX_NGRAM];                // x_{t-k}, k < ngram_max
    int table[kMaxCluster][PLDP_MAX_NGRAM + 1];    // every CTA's cnt[], read over DSMEM
    int warp_tot[kWarps];
    int nstar, offset, mine;
};

// Length of the common suffix of x[0..j] and x[0..t] (x_j == x_t already known),
// capped at n_max.  j < t, so x_{t-m} exists whenever x_{j-m} does.
__device__ __forceinline__ int suffix_match(const int32_t* row, int64_t j, const int32_t* sfx,
                                            int n_max) {
    int m = 1;
    while (m < n_max && j - m >= 0 && __ldg(row + j - m) == sfx[m]) ++m;
    return m;
}

__device__ __forceinline__ void count_hit(int (&c)[PLDP_MAX_NGRAM], int m) {
#pragma unroll
    for (int k = 0; k < PLDP_MAX_NGRAM; ++k) c[k] += (k < m) ? 1 : 0;
}

__device__ __forceinline__ void cluster_arrive() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

template <bool VEC>
__global__ void __launch_bounds__(kThreads)
find_candidates_kernel(const int32_t* __restrict__ ids, int64_t ids_stride,
                       const int32_t* __restrict__ seq_len, int64_t T_cap, int ngram_min,
                       int ngram_max, int32_t* __restrict__ cand_pos, int C_cap,
                       int32_t* __restrict__ cand_count, int32_t* __restrict__ match_len,
                       uint32_t* __restrict__ status, int64_t chunk) {
    __shared__ FindShared sh;
    cg::cluster_group cluster = cg::this_cluster();
    const int CL = static_cast<int>(cluster.num_blocks());
    const int rank = static_cast<int>(cluster.block_rank());
    const int b = blockIdx.x / CL;
    const int tid = threadIdx.x;
    const int lane = tid & 31, warp = tid >> 5;

    // Every CTA of the cluster sees the same seq_len, so these exits are
    // cluster-uniform and no CTA is left waiting at a cluster barrier.
    const int64_t L = seq_len[b];
    if (L < 0 || L > T_cap) {
        if (rank == 0 && tid == 0) {
            cand_count[b] = 0;
            match_len[b] = 0;
            if (status) status[b] |= PLDP_ST_SEQ_LEN;
        }
        return;
    }
    const int64_t t = L - 1;
    if (t < 1) {
        if (rank == 0 && tid == 0) {
            cand_count[b] = 0;
            match_len[b] = 0;
        }
        return;
    }

    const int32_t* row = ids + static_cast<int64_t>(b) * ids_stride;
    if (tid <= PLDP_MAX_NGRAM) sh.cnt[tid] = 0;
    if (tid < ngram_max) sh.suffix[tid] = (t - tid >= 0) ? row[t - tid] : 0;
    __syncthreads();
    const int32_t xt = sh.suffix[0];

    const int64_t c0 = static_cast<int64_t>(rank) * chunk;      // multiple of 4
    const int64_t c1 = min(c0 + chunk, t);                       // scan [c0, c1), all < t

    // ---------------- pass 1: count matches per n-gram length ----------------
    int c[PLDP_MAX_NGRAM];
#pragma unroll
    for (int k = 0; k < PLDP_MAX_NGRAM; ++k) c[k] = 0;

    if (c0 < c1) {
        if constexpr (VEC) {
            const int4* row4 = reinterpret_cast<const int4*>(row);
            const int64_t q0 = c0 >> 2, q1 = (c1 + 3) >> 2;
            for (int64_t qb = q0 + tid; qb < q1; qb += static_cast<int64_t>(kThreads) * kUnroll) {
                int4 v[kUnroll];
#pragma unroll
                for (int u = 0; u < kUnroll; ++u) {
                    const int64_t q = qb + static_cast<int64_t>(u) * kThreads;
                    if (q < q1) v[u] = __ldg(row4 + q);
                }
#pragma unroll
                for (int u = 0; u < kUnroll; ++u) {
                    const int64_t q = qb + static_cast<int64_t>(u) * kThreads;
                    if (q >= q1) continue;
                    const int32_t e[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const int64_t p = 4 * q + k;
                        if (e[k] == xt && p < c1) count_hit(c, suffix_match(row, p, sh.suffix, ngram_max));
                    }
                }
            }
        } else {
            for (int64_t pb = c0 + tid; pb < c1; pb += static_cast<int64_t>(kThreads) * kUnroll) {
                int32_t v[kUnroll];
#pragma unroll
                for (int u = 0; u < kUnroll; ++u) {
                    const int64_t p = pb + static_cast<int64_t>(u) * kThreads;
                    if (p < c1) v[u] = __ldg(row + p);
                }
#pragma unroll
                for (int u = 0; u < kUnroll; ++u) {
                    const int64_t p = pb + static_cast<int64_t>(u) * kThreads;
                    if (p < c1 && v[u] == xt) count_hit(c, suffix_match(row, p, sh.suffix, ngram_max));
                }
            }
        }
    }
#pragma unroll
    for (int k = 0; k < PLDP_MAX_NGRAM; ++k) {
        if (k < ngram_max) {
            const int s = __reduce_add_sync(0xFFFFFFFFu, c[k]);
            if (lane == 0 && s) atomicAdd(&sh.cnt[k + 1], s);
        }
    }

    // ---------------- exchange counts across the cluster ----------------
    cluster.sync();   // every CTA's sh.cnt is final and visible cluster-wide
    for (int i = tid; i < CL * (PLDP_MAX_NGRAM + 1); i += kThreads) {
        const int r = i / (PLDP_MAX_NGRAM + 1), n = i % (PLDP_MAX_NGRAM + 1);
        const int* remote = cluster.map_shared_rank(&sh.cnt[0], r);
        sh.table[r][n] = remote[n];
    }
    __syncthreads();
    cluster_arrive();   // done reading remote shared memory; waited for before exit

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
        sh.offset = off;
        sh.mine = nstar ? sh.table[rank][nstar] : 0;
        if (rank == 0) {
            cand_count[b] = total;
            match_len[b] = nstar;
            if (status && total > C_cap) status[b] |= PLDP_ST_CAND_OVERFLOW;
        }
    }
    __syncthreads();
    const int nstar = sh.nstar, mine = sh.mine;
    int64_t out = sh.offset;

    // ---------------- pass 2: write this CTA's matches in order ----------------
    if (nstar > 0 && mine > 0 && out < C_cap) {
        int32_t* dst = cand_pos + static_cast<int64_t>(b) * C_cap;
        const int64_t end = out + mine;
        constexpr int G = VEC ? 4 : 1;                       // positions per thread per tile
        const int64_t g0 = c0 / G, g1 = (c1 + G - 1) / G;
        for (int64_t gb = g0; gb < g1 && out < end && out < C_cap; gb += kThreads) {
            const int64_t g = gb + tid;
            uint32_t mask = 0;
            if (g < g1) {
                int32_t e[G];
                if constexpr (VEC) {
                    const int4 v = __ldg(reinterpret_cast<const int4*>(row) + g);
                    e[0] = v.x; e[1] = v.y; e[2] = v.z; e[3] = v.w;
                } else {
                    e[0] = __ldg(row + g);
                }
#pragma unroll
                for (int k = 0; k < G; ++k) {
                    const int64_t p = g * G + k;
                    if (e[k] == xt && p < c1 && suffix_match(row, p, sh.suffix, ngram_max) >= nstar)
                        mask |= 1u << k;
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
            for (int w = 0; w < kWarps; ++w) {
                const int x = sh.warp_tot[w];
                before += (w < warp) ? x : 0;
                tile += x;
            }
            int64_t pos = out + before + (incl - cnt);
            while (mask) {
                const int k = __ffs(mask) - 1;
                mask &= mask - 1;
                if (pos < C_cap) dst[pos] = static_cast<int32_t>(g * G + k);
                ++pos;
            }
            out += tile;
            __syncthreads();   // warp_tot is rewritten by the next tile
        }
    }
    cluster_wait();   // no CTA leaves while another may still read its shared memory
}

}  // namespace
}  // namespace pldp

using namespace pldp;

extern "C" PLDP_API pldp_status pldp_find_candidates(const int32_t* ids, int64_t ids_stride,
                                                     const int32_t* seq_len, int B, int64_t T_cap,
                                                     int ngram_min, int ngram_max,
                                                     int32_t* cand_pos, int C_cap,
                                                     int32_t* cand_count, int32_t* match_len,
                                                     uint32_t* status, void* stream) {
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "find_candidates: B < 0");
    if (T_cap < 0 || T_cap > INT32_MAX)
        return fail(PLDP_ERR_INVALID_ARG, "find_candidates: T_cap outside [0, 2^31)");
    if (ids_stride < T_cap) return fail(PLDP_ERR_INVALID_ARG, "find_candidates: ids_stride < T_cap");
    if (ngram_min < 1 || ngram_max < ngram_min || ngram_max > PLDP_MAX_NGRAM)
        return fail(PLDP_ERR_INVALID_ARG, "find_candidates: need 1 <= ngram_min <= ngram_max <= %d",
                    PLDP_MAX_NGRAM);
    if (C_cap < 0) return fail(PLDP_ERR_INVALID_ARG, "find_candidates: C_cap < 0");
    if (B == 0) return PLDP_OK;
    if (!ids || !seq_len || !cand_count || !match_len || (C_cap > 0 && !cand_pos))
        return fail(PLDP_ERR_INVALID_ARG, "find_candidates: null pointer");

    const bool vec = aligned16(ids) && ids_stride % 4 == 0 && T_cap % 4 == 0;
    // One CTA per kPositionsPerCta positions, at most a portable cluster, and no
    // more CTAs in all than fit on the device at once (a single wave).
    int CL = static_cast<int>((T_cap + kPositionsPerCta - 1) / kPositionsPerCta);
    const void* fn = vec ? reinterpret_cast<const void*>(&find_candidates_kernel<true>)
                         : reinterpret_cast<const void*>(&find_candidates_kernel<false>);
    const int per_seq = resident_blocks(fn, kThreads, 0) / B;
    if (CL > per_seq) CL = per_seq;
    CL = CL < 1 ? 1 : (CL > kMaxCluster ? kMaxCluster : CL);
    int64_t chunk = (T_cap + CL - 1) / CL;
    chunk = (chunk + 3) / 4 * 4;
    if (chunk < 4) chunk = 4;
    if (static_cast<int64_t>(B) * CL > INT32_MAX)
        return fail(PLDP_ERR_INVALID_ARG, "find_candidates: B too large");

    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(B * CL));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = static_cast<cudaStream_t>(stream);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CL;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e;
    if (vec)
        e = cudaLaunchKernelEx(&cfg, find_candidates_kernel<true>, ids, ids_stride, seq_len, T_cap,
                               ngram_min, ngram_max, cand_pos, C_cap, cand_count, match_len, status,
                               chunk);
    else
        e = cudaLaunchKernelEx(&cfg, find_candidates_kernel<false>, ids, ids_stride, seq_len, T_cap,
                               ngram_min, ngram_max, cand_pos, C_cap, cand_count, match_len, status,
                               chunk);
    if (e != cudaSuccess)
        return fail(PLDP_ERR_CUDA, "find_candidates: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}
