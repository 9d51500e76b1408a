// pldp_find_candidates: the candidate search of PLD+ (Eq. 1, Sec. 4.2, with the
// longest-suffix n-gram rule) as its own kernel -- one thread-block cluster per
// sequence running the scan of pldp_scan.cuh.
#include "pldp_scan.cuh"

namespace pldp {
namespace {

constexpr int64_t kPositionsPerCta = 4096;

template <bool VEC>
__global__ void __launch_bounds__(kScanThreads)
find_candidates_kernel(const int32_t* __restrict__ ids, int64_t ids_stride,
                       const int32_t* __restrict__ seq_len, int64_t T_cap, int ngram_min,
                       int ngram_max, int32_t* __restrict__ cand_pos, int C_cap,
                       int32_t* __restrict__ cand_count, int32_t* __restrict__ match_len,
                       uint32_t* __restrict__ status, int64_t chunk) {
    __shared__ ScanShared sh;
    pdl_enter();
    cg::cluster_group cluster = cg::this_cluster();
    const int CL = static_cast<int>(cluster.num_blocks());
    const int rank = static_cast<int>(cluster.block_rank());
    const int b = blockIdx.x / CL;
    const int tid = threadIdx.x;

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
    const int64_t c0 = static_cast<int64_t>(rank) * chunk;
    const int64_t c1 = min(c0 + chunk, t);
    int c[PLDP_MAX_NGRAM];
#pragma unroll
    for (int k = 0; k < PLDP_MAX_NGRAM; ++k) c[k] = 0;
    const GlobalIds src{row};
    scan_count<VEC>(src, row, c0, c1, t, ngram_max, c);
    __syncthreads();                       // sh.cnt zeroed before the adds
    scan_reduce_counts(c, ngram_max, sh);

    cluster.sync();                        // every CTA's counts are final
    scan_decide(cluster, sh, CL, rank, ngram_min, ngram_max);
    cluster_arrive();                      // remote reads done; waited for before exit
    if (rank == 0 && tid == 0) {
        cand_count[b] = sh.total;
        match_len[b] = sh.nstar;
        if (status && sh.total > C_cap) status[b] |= PLDP_ST_CAND_OVERFLOW;
    }
    scan_write<VEC>(src, row, c0, c1, t, ngram_max, sh, cand_pos + static_cast<int64_t>(b) * C_cap, C_cap);
    cluster_wait();
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
    const void* fn = vec ? reinterpret_cast<const void*>(&find_candidates_kernel<true>)
                         : reinterpret_cast<const void*>(&find_candidates_kernel<false>);
    int CL;
    int64_t chunk;
    scan_shape(T_cap, B, resident_blocks(fn, kScanThreads, 0), kPositionsPerCta, &CL, &chunk);
    if (static_cast<int64_t>(B) * CL > INT32_MAX)
        return fail(PLDP_ERR_INVALID_ARG, "find_candidates: B too large");

    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(B * CL));
    cfg.blockDim = dim3(kScanThreads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = static_cast<cudaStream_t>(stream);
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CL;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
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
