// Induction-head identification (Sec. 4.2.1): an offline utility that picks the
// attention rows (layer, head) that Eq. 2 aggregates.  For a generated token x_p
// that also occurs earlier, the position r* it was most likely copied from is
// the occurrence whose preceding tokens match the output's longest; a row
// "points at" r* when its attention of query p-1 is largest at key r*.  Counting
// that over many observations and keeping the rows with the most counts gives
// G* x L*.
//
// pldp_identify_heads: a (group of kRowsPerCta rows, observation) grid of CTAs.
//  1. The context before x_p is scanned for x_p, each cluster of up to 8 CTAs of
//     the observation splitting it into consecutive parts (4 bytes per position
//     against 2 R bytes of attention); every occurrence j gets its overlap ov(j)
//     (the length of the common suffix of x[..j] and x[..p], measured by the whole
//     warp, 32 offsets per round trip) and r* = argmax ov, the smaller j on ties,
//     from a max of packed keys (ov << 32 | ~j) over the CTA and then over the
//     cluster: each CTA writes its key into every peer's shared memory and arrives
//     on the cluster barrier.
//  2. The R rows of query p-1 are reduced to their first maximum, one warp per
//     row (16-byte streaming loads where rows allow, packed (value, ~key)
//     maxima).  Only then does the CTA wait on the cluster barrier -- its peers'
//     keys arrived long before -- and a row whose maximum is at r* adds one to
//     counts[r].  The short latency-bound scan thus comes first and the rows
//     (the bandwidth) after it, and no CTA waits at its end for a slower peer or
//     stays resident for peers that still read its shared memory.
// pldp_top_heads: one CTA ranks the counts and writes the k rows with the most
// (ties to the smaller row index) -- the row_idx of pldp_rank_attention.
#include "pldp_internal.cuh"

namespace pldp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxTopRows = 8192;   // counts staged in shared memory by pldp_top_heads
constexpr int kRowsPerCta = 8;      // attention rows per CTA (one per warp)
constexpr int kIdentCluster = 8;    // CTAs of one observation that share its copy-source scan

// The first maximum of elements [0, n) of one attention row, by one warp, as a
// packed (value, ~key) key.  Each lane keeps a running (max, first key) over its
// vectors in increasing key order, and packs once.
template <typename T>
__device__ __forceinline__ unsigned long long row_first_max_vec(const T* row, int64_t n, int lane) {
    constexpr int VW = 16 / static_cast<int>(sizeof(T));
    const int64_t nv = n / VW;
    const uint4* p = reinterpret_cast<const uint4*>(row);
    float bv = -INFINITY;
    int64_t bi = -1;
    for (int64_t v0 = lane; v0 < nv; v0 += 32 * 8) {
        uint4 x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
            if (v0 + 32 * u < nv) x[u] = ld_stream16(p + v0 + 32 * u);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            if (v0 + 32 * u >= nv) continue;
            const float m = vmax(x[u], T());
            if (m > bv || bi < 0) {
                bv = m;
                bi = (v0 + 32 * u) * VW + vfirst(x[u], m, T());
            }
        }
    }
    for (int64_t k = nv * VW + lane; k < n; k += 32) {              // the tail
        const float v = to_f32(row[k]);
        if (v > bv || bi < 0) {
            bv = v;
            bi = k;
        }
    }
    // every lane takes part in the reduction; a lane without elements offers 0 (no key)
    return warp_max_u64(bi < 0 ? 0ull : pack_key(bv, static_cast<uint32_t>(bi)));
}

template <typename T>
__device__ __forceinline__ unsigned long long row_first_max_elem(const T* row, int64_t n, int lane) {
    float bv = -INFINITY;
    int64_t bi = -1;
    for (int64_t k = lane; k < n; k += 32) {
        const float v = to_f32(row[k]);
        if (v > bv || bi < 0) {
            bv = v;
            bi = k;
        }
    }
    // every lane takes part in the reduction; a lane without elements offers 0 (no key)
    return warp_max_u64(bi < 0 ? 0ull : pack_key(bv, static_cast<uint32_t>(bi)));
}

template <bool VEC>
__device__ __forceinline__ unsigned long long row_first_max(const void* row, bool bf16, int64_t n, int lane) {
    if (VEC)
        return bf16 ? row_first_max_vec(static_cast<const __nv_bfloat16*>(row), n, lane)
                    : row_first_max_vec(static_cast<const float*>(row), n, lane);
    return bf16 ? row_first_max_elem(static_cast<const __nv_bfloat16*>(row), n, lane)
                : row_first_max_elem(static_cast<const float*>(row), n, lane);
}

// Packed (ov, ~j) key of occurrence j of x_p (x_j = x_p known), by the whole warp
// (j, p warp-uniform): lane k of a round compares x_{j-k} with x_{p-k}, so the
// common suffix is measured 32 tokens per round trip instead of one, and ov is
// the first offset that differs (or max_suffix, or j + 1 at the context start).
__device__ __forceinline__ unsigned long long warp_occurrence_key(const int32_t* __restrict__ x, int64_t j,
                                                                  int64_t p, int max_suffix, int lane) {
    int ov = max_suffix;
    for (int k0 = 0; k0 < max_suffix; k0 += 32) {
        const int k = k0 + lane;
        const bool same = k < max_suffix && j - k >= 0 && __ldg(x + j - k) == __ldg(x + p - k);
        const unsigned diff = __ballot_sync(0xFFFFFFFFu, !same);
        if (diff) {                                                 // warp-uniform
            ov = k0 + __ffs(diff) - 1;
            break;
        }
    }
    return (static_cast<unsigned long long>(ov) << 32) |
           static_cast<unsigned long long>(0xFFFFFFFFu - static_cast<uint32_t>(j));
}

// The occurrences a warp found in one tile, walked by the whole warp one at a time:
// lane L's bit i of `hits` stands for position pos_of(L, i).  Every lane runs every
// iteration (the loop condition is a ballot).
template <typename PosOf>
__device__ __forceinline__ void walk_hits(uint32_t hits, const int32_t* __restrict__ x, int64_t p, int max_suffix,
                                          int lane, unsigned long long& best, PosOf pos_of) {
    for (unsigned who = __ballot_sync(0xFFFFFFFFu, hits != 0); who; who = __ballot_sync(0xFFFFFFFFu, hits != 0)) {
        const int L = __ffs(who) - 1;
        const int bit = __shfl_sync(0xFFFFFFFFu, __ffs(hits) - 1, L);
        const unsigned long long key = warp_occurrence_key(x, pos_of(L, bit), p, max_suffix, lane);
        best = key > best ? key : best;
        if (lane == L) hits &= hits - 1;
    }
}

template <bool VEC, bool IVEC>
__global__ void __launch_bounds__(kThreads, 4)   // 64 registers: 4 CTAs per SM
identify_heads_kernel(const int32_t* __restrict__ ids, int64_t ids_stride, const int32_t* __restrict__ pos,
                      int64_t T_cap, int max_suffix, const void* __restrict__ A, bool a_bf16, int R,
                      int64_t row_stride, int64_t seq_stride, unsigned* __restrict__ counts,
                      int32_t* __restrict__ r_star, uint32_t* __restrict__ status) {
    __shared__ unsigned long long wkey[kWarps];
    __shared__ unsigned long long peer_key[kIdentCluster];        // the best occurrence key of each CTA of the cluster
    pdl_enter();
    const int b = blockIdx.y;                                     // the CTAs of one observation are adjacent:
    const int r0 = blockIdx.x * kRowsPerCta;                      // its ids are read once from DRAM, then L2
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t p = pos[b];
    if (p < 1 || p >= T_cap) {
        if (tid == 0 && blockIdx.x == 0) {
            if (r_star) r_star[b] = -1;
            if (status) atomicOr(status + b, PLDP_ST_SEQ_LEN);
        }
        return;
    }
    const int32_t* x = ids + static_cast<int64_t>(b) * ids_stride;
    const int32_t xp = __ldg(x + p);
    // every CTA of the cluster must be running before any writes into its shared memory
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    // 1. the copy source r*: the cluster's CTAs (those of one observation) scan
    //    consecutive parts of [0, p) in tiles, several loads in flight per thread, and
    //    meet over distributed shared memory
    cg::cluster_group cluster = cg::this_cluster();
    const int64_t cs = static_cast<int64_t>(cluster.num_blocks()), crank = cluster.block_rank();
    unsigned long long best = 0;
    constexpr int U = IVEC ? 4 : 8;                         // loads in flight per thread
    // Tiles are walked per warp (the loop bounds are warp-uniform) so that each
    // warp's occurrences can be measured by all its lanes together.
    const int64_t wbase = static_cast<int64_t>(warp) * 32;
    if constexpr (IVEC) {
        static_assert(U * 4 <= 32, "one hit bit per position of a tile");
        const int4* x4 = reinterpret_cast<const int4*>(x);
        const int64_t nq = (p + 3) / 4;                             // int4 units covering [0, p)
        const int64_t q_lo = nq * crank / cs, q_hi = nq * (crank + 1) / cs;
        for (int64_t qb = q_lo + wbase; qb < q_hi; qb += static_cast<int64_t>(kThreads) * U) {
            const int64_t q0 = qb + lane;
            int4 v[U];
#pragma unroll
            for (int u = 0; u < U; ++u)
                if (q0 + u * kThreads < q_hi) v[u] = __ldg(x4 + q0 + u * kThreads);
            uint32_t hits = 0;
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int64_t q = q0 + u * kThreads;
                if (q >= q_hi) continue;
                const int32_t e[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    if (4 * q + c < p && e[c] == xp) hits |= 1u << (4 * u + c);
            }
            walk_hits(hits, x, p, max_suffix, lane, best, [&](int L, int bit) {
                return 4 * (qb + L + static_cast<int64_t>(bit >> 2) * kThreads) + (bit & 3);
            });
        }
    } else {
        const int64_t j_lo = p * crank / cs, j_hi = p * (crank + 1) / cs;
        for (int64_t jb = j_lo + wbase; jb < j_hi; jb += static_cast<int64_t>(kThreads) * U) {
            const int64_t j0 = jb + lane;
            int32_t v[U];
#pragma unroll
            for (int u = 0; u < U; ++u)
                if (j0 + u * kThreads < j_hi) v[u] = __ldg(x + j0 + u * kThreads);
            uint32_t hits = 0;
#pragma unroll
            for (int u = 0; u < U; ++u)
                if (j0 + u * kThreads < j_hi && v[u] == xp) hits |= 1u << u;
            walk_hits(hits, x, p, max_suffix, lane, best, [&](int L, int bit) {
                return jb + L + static_cast<int64_t>(bit) * kThreads;
            });
        }
    }
    best = warp_max_u64(best);
    if (lane == 0) wkey[warp] = best;
    asm volatile("barrier.cluster.wait.aligned;" ::: "memory");  // every peer has started
    __syncthreads();
    if (tid == 0) {                                               // this CTA's best, into every peer's slot
        unsigned long long k = 0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) k = wkey[w] > k ? wkey[w] : k;
        for (int c = 0; c < static_cast<int>(cs); ++c) *cluster.map_shared_rank(&peer_key[crank], c) = k;
    }
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
    // 2. the first maximum of each of this CTA's rows, one row per warp, while the
    //    peers' keys come in
    constexpr int RW = kRowsPerCta / kWarps;
    const size_t es = a_bf16 ? 2 : 4;
    const char* ab = static_cast<const char*>(A) + static_cast<int64_t>(b) * seq_stride * es;
    const int r1 = r0 + kRowsPerCta < R ? r0 + kRowsPerCta : R;
    unsigned long long rk[RW];
#pragma unroll
    for (int i = 0; i < RW; ++i) {
        const int r = r0 + warp + i * kWarps;
        rk[i] = r < r1 ? row_first_max<VEC>(ab + static_cast<int64_t>(r) * row_stride * es, a_bf16, p, lane) : 0ull;
    }
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");   // every peer's key is in
    best = 0;
    for (int c = 0; c < static_cast<int>(cs); ++c) best = peer_key[c] > best ? peer_key[c] : best;
    const int64_t rs = best ? static_cast<int64_t>(0xFFFFFFFFu - static_cast<uint32_t>(best & 0xFFFFFFFFull)) : -1;
    if (tid == 0 && blockIdx.x == 0 && r_star) r_star[b] = static_cast<int32_t>(rs);
    if (rs < 0) return;
    // the rows whose maximum is at r* count
#pragma unroll
    for (int i = 0; i < RW; ++i) {
        const int r = r0 + warp + i * kWarps;
        if (lane == 0 && r < r1 && rk[i] && static_cast<int64_t>(key_index(rk[i])) == rs) atomicAdd(counts + r, 1u);
    }
}

// The k rows with the most counts, ties to the smaller row: a row's rank is the
// number of rows that beat it.
__global__ void __launch_bounds__(1024) top_heads_kernel(const unsigned* __restrict__ counts, int R, int k,
                                                         int32_t* __restrict__ row_idx) {
    __shared__ unsigned c[kMaxTopRows];
    pdl_enter();
    for (int r = threadIdx.x; r < R; r += blockDim.x) c[r] = counts[r];
    __syncthreads();
    for (int r = threadIdx.x; r < R; r += blockDim.x) {
        const unsigned mine = c[r];
        int rank = 0;
        for (int q = 0; q < R; ++q) rank += (c[q] > mine || (c[q] == mine && q < r)) ? 1 : 0;
        if (rank < k) row_idx[rank] = r;
    }
}

}  // namespace
}  // namespace pldp

using namespace pldp;

extern "C" PLDP_API pldp_status pldp_identify_heads(const int32_t* ids, int64_t ids_stride, const int32_t* pos,
                                                    int B, int64_t T_cap, int max_suffix, const void* A,
                                                    pldp_dtype dtype, int R, int64_t row_stride,
                                                    int64_t seq_stride, uint32_t* counts, int32_t* r_star,
                                                    uint32_t* status, void* stream) {
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "identify_heads: B < 0");
    if (dtype != PLDP_F32 && dtype != PLDP_BF16)
        return fail(PLDP_ERR_UNSUPPORTED, "identify_heads: unsupported dtype %d", (int)dtype);
    if (R < 1) return fail(PLDP_ERR_INVALID_ARG, "identify_heads: R < 1");
    if (max_suffix < 1) return fail(PLDP_ERR_INVALID_ARG, "identify_heads: max_suffix < 1");
    if (T_cap < 0 || T_cap > INT32_MAX) return fail(PLDP_ERR_INVALID_ARG, "identify_heads: bad T_cap");
    if (ids_stride < T_cap) return fail(PLDP_ERR_INVALID_ARG, "identify_heads: ids_stride < T_cap");
    if (row_stride < T_cap) return fail(PLDP_ERR_INVALID_ARG, "identify_heads: row_stride < T_cap");
    if (seq_stride < static_cast<int64_t>(R) * row_stride)
        return fail(PLDP_ERR_INVALID_ARG, "identify_heads: seq_stride < R*row_stride");
    if (B > 65535) return fail(PLDP_ERR_UNSUPPORTED, "identify_heads: B > 65535");
    if (B == 0) return PLDP_OK;
    if (!ids || !pos || !A || !counts) return fail(PLDP_ERR_INVALID_ARG, "identify_heads: null pointer");
    const size_t es = dtype == PLDP_F32 ? 4 : 2;
    const bool vec = aligned16(A) && (row_stride * es) % 16 == 0 && (seq_stride * es) % 16 == 0;
    const bool bf16 = dtype == PLDP_BF16;
    const bool ivec = aligned16(ids) && ids_stride % 4 == 0;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // the CTAs of an observation in clusters of up to kIdentCluster (the grid padded to a
    // whole number of them; padding CTAs hold no rows and only scan)
    const int groups = (R + kRowsPerCta - 1) / kRowsPerCta;
    const int cs = groups < kIdentCluster ? groups : kIdentCluster;
    const dim3 grid(static_cast<unsigned>((groups + cs - 1) / cs * cs), static_cast<unsigned>(B));
    cudaError_t e;
#define PLDP_IDENTIFY_LAUNCH(V, I)                                                                          \
    launch_pdl(identify_heads_kernel<V, I>, grid, dim3(kThreads), 0, s, cs, ids, ids_stride, pos, T_cap, max_suffix, \
               A, bf16, R, row_stride, seq_stride, static_cast<unsigned*>(counts), r_star, status)
    if (vec)
        e = ivec ? PLDP_IDENTIFY_LAUNCH(true, true) : PLDP_IDENTIFY_LAUNCH(true, false);
    else
        e = ivec ? PLDP_IDENTIFY_LAUNCH(false, true) : PLDP_IDENTIFY_LAUNCH(false, false);
#undef PLDP_IDENTIFY_LAUNCH
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "identify_heads: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}

extern "C" PLDP_API pldp_status pldp_top_heads(const uint32_t* counts, int R, int k, int32_t* row_idx,
                                               void* stream) {
    if (R < 1 || R > kMaxTopRows) return fail(PLDP_ERR_INVALID_ARG, "top_heads: need 1 <= R <= %d", kMaxTopRows);
    if (k < 1 || k > R) return fail(PLDP_ERR_INVALID_ARG, "top_heads: need 1 <= k <= R");
    if (!counts || !row_idx) return fail(PLDP_ERR_INVALID_ARG, "top_heads: null pointer");
    const cudaError_t e = launch_pdl(top_heads_kernel, dim3(1), dim3(1024), 0, static_cast<cudaStream_t>(stream), 0,
                                     static_cast<const unsigned*>(counts), R, k, row_idx);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "top_heads: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}
