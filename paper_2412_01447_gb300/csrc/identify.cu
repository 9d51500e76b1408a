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
//     (the length of the common suffix of x[..j] and x[..p]) and r* = argmax ov,
//     the smaller j on ties, from a max of packed keys (ov << 32 | ~j) over the
//     CTA and then over the cluster's distributed shared memory.
//  2. The R rows of query p-1 are reduced to their first maximum, one warp per
//     row (16-byte streaming loads where rows allow, packed (value, ~key)
//     maxima), and a row whose maximum is at r* adds one to counts[r].  The rows
//     are read first (they do not depend on r*, and they are the bandwidth); the
//     latency-bound scan of step 1 follows.
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

// Packed (ov, ~j) key of occurrence j of x_p (x_j = x_p known), or 0.
__device__ __forceinline__ unsigned long long occurrence_key(const int32_t* __restrict__ x, int64_t j, int64_t p,
                                                             int max_suffix) {
    int k = 1;                                                      // x_j = x_p itself
    while (k < max_suffix && j - k >= 0 && __ldg(x + j - k) == __ldg(x + p - k)) ++k;
    return (static_cast<unsigned long long>(k) << 32) |
           static_cast<unsigned long long>(0xFFFFFFFFu - static_cast<uint32_t>(j));
}

template <bool VEC, bool IVEC>
__global__ void __launch_bounds__(kThreads)
identify_heads_kernel(const int32_t* __restrict__ ids, int64_t ids_stride, const int32_t* __restrict__ pos,
                      int64_t T_cap, int max_suffix, const void* __restrict__ A, bool a_bf16, int R,
                      int64_t row_stride, int64_t seq_stride, unsigned* __restrict__ counts,
                      int32_t* __restrict__ r_star, uint32_t* __restrict__ status) {
    __shared__ unsigned long long wkey[kWarps];
    __shared__ unsigned long long cta_key;                        // this CTA's best occurrence key
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
    // 2 (first: it does not depend on r*, and it is the bandwidth). The first maximum of
    // each of this CTA's rows, two rows per warp.
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
    // 1. the copy source r*: the cluster's CTAs (those of one observation) scan
    //    consecutive parts of [0, p) in tiles, eight loads in flight per thread, and
    //    meet over distributed shared memory
    cg::cluster_group cluster = cg::this_cluster();
    const int64_t cs = static_cast<int64_t>(cluster.num_blocks()), crank = cluster.block_rank();
    unsigned long long best = 0;
    constexpr int U = 8;
    if constexpr (IVEC) {
        const int4* x4 = reinterpret_cast<const int4*>(x);
        const int64_t nq = (p + 3) / 4;                             // int4 units covering [0, p)
        const int64_t q_lo = nq * crank / cs, q_hi = nq * (crank + 1) / cs;
        for (int64_t q0 = q_lo + tid; q0 < q_hi; q0 += static_cast<int64_t>(kThreads) * U) {
            int4 v[U];
#pragma unroll
            for (int u = 0; u < U; ++u)
                if (q0 + u * kThreads < q_hi) v[u] = __ldg(x4 + q0 + u * kThreads);
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int64_t q = q0 + u * kThreads;
                if (q >= q_hi) continue;
                const int32_t e[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    const int64_t j = 4 * q + c;
                    if (j < p && e[c] == xp) {
                        const unsigned long long key = occurrence_key(x, j, p, max_suffix);
                        best = key > best ? key : best;
                    }
                }
            }
        }
    } else {
        const int64_t j_lo = p * crank / cs, j_hi = p * (crank + 1) / cs;
        for (int64_t j0 = j_lo + tid; j0 < j_hi; j0 += static_cast<int64_t>(kThreads) * U) {
            int32_t v[U];
#pragma unroll
            for (int u = 0; u < U; ++u)
                if (j0 + u * kThreads < j_hi) v[u] = __ldg(x + j0 + u * kThreads);
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int64_t j = j0 + u * kThreads;
                if (j < j_hi && v[u] == xp) {
                    const unsigned long long key = occurrence_key(x, j, p, max_suffix);
                    best = key > best ? key : best;
                }
            }
        }
    }
    best = warp_max_u64(best);
    if (lane == 0) wkey[warp] = best;
    __syncthreads();
    if (tid == 0) {
        unsigned long long k = 0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) k = wkey[w] > k ? wkey[w] : k;
        cta_key = k;
    }
    cluster.sync();                                               // every CTA's part is in
    if (tid == 0) {
        unsigned long long k = 0;
        for (int c = 0; c < static_cast<int>(cs); ++c) {
            const unsigned long long o = *cluster.map_shared_rank(&cta_key, c);
            k = o > k ? o : k;
        }
        wkey[0] = k;
    }
    cluster.sync();                                               // read before any CTA of the cluster leaves
    best = wkey[0];
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
