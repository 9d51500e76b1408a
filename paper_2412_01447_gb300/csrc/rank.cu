// Candidate ranking of PLD+:
//   hidden states -- Eq. 3 (Sec. 4.2.2): j* = argmax_{j in P} cos(H_{j-1}, H_{t-1})
//   attentions    -- Eq. 2 (Sec. 4.2.1): j* = argmax_{j in P} max_{(l,g) in L* x G*} A^{(l,g)}_{t-1}[j]
//
// One thread-block cluster per sequence; candidates are dealt round-robin over
// the cluster's CTAs and then over their warps, one candidate per warp at a
// time.  Each CTA reduces its warps' packed (score, position) keys, and CTA 0
// of the cluster reduces the CTAs' keys over distributed shared memory.  The
// packed key makes the argmax independent of reduction order: the larger
// score wins, equal scores go to the smaller position.
//
// Hidden ranking stages the query row H_{t-1} in shared memory with one bulk
// asynchronous copy (when rows are 16-byte aligned) issued before the warps
// start streaming their candidate rows, so the two DRAM round trips overlap.
#include <math.h>

#include "pldp_internal.cuh"

namespace pldp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxCluster = 8;
constexpr int kRowUnroll = 8;                 // 16-byte loads in flight per lane
constexpr size_t kMaxQueryBytes = 196608;     // d * sizeof(dtype) limit
constexpr int kMaxSelRows = 8192;             // row_idx entries staged in shared memory

__device__ __forceinline__ void cl_arrive() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cl_wait() {
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

struct ArgmaxShared {
    unsigned long long warp_key[kWarps];
    unsigned long long cta_key;
    int cta_err;
    int warp_err[kWarps];
};

// Reduces the per-warp keys (set by lane 0 of every warp) to the cluster's best
// and writes it out from CTA 0.  Must be reached by every thread of every CTA.
__device__ __forceinline__ void cluster_argmax_store(cg::cluster_group& cluster, ArgmaxShared& sh,
                                                     int b, int32_t* best_pos, float* best_score,
                                                     uint32_t* status, uint32_t err_bit) {
    const int tid = threadIdx.x;
    __syncthreads();
    if (tid == 0) {
        unsigned long long k = 0;
        int err = 0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
            k = sh.warp_key[w] > k ? sh.warp_key[w] : k;
            err |= sh.warp_err[w];
        }
        sh.cta_key = k;
        sh.cta_err = err;
    }
    cluster.sync();
    if (cluster.block_rank() == 0 && tid < 32) {
        const int CL = static_cast<int>(cluster.num_blocks());
        unsigned long long k = 0;
        int err = 0;
        if (tid < CL) {
            ArgmaxShared* remote = cluster.map_shared_rank(&sh, tid);
            k = remote->cta_key;
            err = remote->cta_err;
        }
        k = warp_max_u64(k);
        err = __reduce_or_sync(0xFFFFFFFFu, err);
        if (tid == 0) {
            if (err) {
                best_pos[b] = -1;
                if (best_score) best_score[b] = -INFINITY;
                if (status) status[b] |= err_bit;
            } else if (k == 0) {
                best_pos[b] = -1;
                if (best_score) best_score[b] = -INFINITY;
            } else {
                best_pos[b] = static_cast<int32_t>(key_index(k));
                if (best_score) best_score[b] = key_value(k);
            }
        }
    }
    cl_arrive();
    cl_wait();   // CTA 0 has read every CTA's shared memory before any exits
}

// ---------------------------------------------------------------------------
// hidden-state ranking
// ---------------------------------------------------------------------------
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
__device__ __forceinline__ float finish_cosine(float dot, float na, float nq) {
    if (na == 0.0f || nq == 0.0f) return 0.0f;
    return static_cast<float>(static_cast<double>(dot) /
                              sqrt(static_cast<double>(na) * static_cast<double>(nq)));
}

template <typename T, bool VEC>
__global__ void __launch_bounds__(kThreads)
rank_hidden_kernel(const T* __restrict__ H, int64_t d, int64_t seq_stride,
                   const int32_t* __restrict__ seq_len, int64_t T_cap,
                   const int32_t* __restrict__ cand_pos, const int32_t* __restrict__ cand_count,
                   int C_cap, float threshold, float* __restrict__ scores,
                   int32_t* __restrict__ best_pos, float* __restrict__ best_score,
                   uint32_t* __restrict__ status) {
    extern __shared__ __align__(128) unsigned char dyn_smem[];
    T* q_sh = reinterpret_cast<T*>(dyn_smem);          // query row H_{t-1}
    __shared__ ArgmaxShared sh;
    __shared__ __align__(8) uint64_t bar;

    cg::cluster_group cluster = cg::this_cluster();
    const int CL = static_cast<int>(cluster.num_blocks());
    const int rank = static_cast<int>(cluster.block_rank());
    const int b = blockIdx.x / CL;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    const int64_t L = seq_len[b];
    if (L < 0 || L > T_cap) {       // cluster-uniform exit
        if (rank == 0 && tid == 0) {
            best_pos[b] = -1;
            if (best_score) best_score[b] = -INFINITY;
            if (status) status[b] |= PLDP_ST_SEQ_LEN;
        }
        return;
    }
    const int64_t t = L - 1;
    int n = cand_count[b];
    n = n < 0 ? 0 : (n > C_cap ? C_cap : n);
    const int stride_cand = CL * kWarps;
    // this CTA owns candidates rank, rank + CL, ...; warp w takes every kWarps-th of those.
    // With t < 2 no candidate is eligible (j >= 1 and j < t), but the listed ones
    // still get their -inf scores written.
    const bool cta_work = rank < n;
    const bool need_query = cta_work && t >= 2;
    const T* hb = H + static_cast<int64_t>(b) * seq_stride;

    if (lane == 0) {
        sh.warp_key[warp] = 0;
        sh.warp_err[warp] = 0;
    }
    bool q_ready = true;
    if (need_query) {
        const T* qg = hb + (t - 1) * d;
        const uint32_t qbytes = static_cast<uint32_t>(d * sizeof(T));
        if constexpr (VEC) {
            if (tid == 0) {
                mbar_init(&bar, 1);
                fence_mbar_init();
            }
            __syncthreads();
            if (tid == 0) {
                mbar_arrive_expect_tx(&bar, qbytes);
                bulk_g2s(q_sh, qg, qbytes, &bar);
            }
            q_ready = false;      // waited for right before the first use
        } else {
            for (int64_t k = tid; k < d; k += kThreads) q_sh[k] = qg[k];
            __syncthreads();
        }
    }

    bool timed_out = false;
    if (cta_work) {
        for (int i = rank + CL * warp; i < n; i += stride_cand) {
            const int64_t j = cand_pos[static_cast<int64_t>(b) * C_cap + i];
            const bool ok = (j >= 1 && j < t);
            float s = -INFINITY;
            if (ok) {
                const T* row = hb + (j - 1) * d;          // H_{j-1}
                float dot = 0.f, na = 0.f, nq = 0.f;
                if constexpr (VEC) {
                    constexpr int E = 16 / sizeof(T);
                    const int64_t nch = d / E;
                    for (int64_t c0 = lane; c0 < nch; c0 += 32 * kRowUnroll) {
                        uint4 a[kRowUnroll];
#pragma unroll
                        for (int u = 0; u < kRowUnroll; ++u) {
                            const int64_t c = c0 + 32 * u;
                            if (c < nch) a[u] = ld_stream16(row + c * E);
                        }
                        if (!q_ready) {
                            if (!mbar_wait(&bar, 0, kMbarPolls)) timed_out = true;
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
                } else {
                    for (int64_t k = lane; k < d; k += 32) {
                        const float x = to_f32(row[k]), y = to_f32(q_sh[k]);
                        dot = fmaf(x, y, dot);
                        na = fmaf(x, x, na);
                        nq = fmaf(y, y, nq);
                    }
                }
                dot = warp_sum(dot);
                na = warp_sum(na);
                nq = warp_sum(nq);
                s = finish_cosine(dot, na, nq);
            }
            if (__any_sync(0xFFFFFFFFu, timed_out)) {
                timed_out = true;
                break;
            }
            if (lane == 0) {
                if (scores) scores[static_cast<int64_t>(b) * C_cap + i] = s;
                if (ok && s > threshold) {
                    const unsigned long long k = pack_key(s, static_cast<uint32_t>(j));
                    if (k > sh.warp_key[warp]) sh.warp_key[warp] = k;
                }
            }
        }
        if constexpr (VEC) {
            // A warp that never consumed the query still makes sure the copy into this
            // CTA's shared memory has landed before the CTA can exit (bounded).
            if (!q_ready && !mbar_wait(&bar, 0, kMbarPolls)) timed_out = true;
        }
        if (lane == 0 && timed_out) sh.warp_err[warp] = 1;
    }
    cluster_argmax_store(cluster, sh, b, best_pos, best_score, status, PLDP_ST_TIMEOUT);
}

// ---------------------------------------------------------------------------
// attention ranking
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(kThreads)
rank_attention_kernel(const T* __restrict__ A, int R, int64_t row_stride, int64_t seq_stride,
                      const int32_t* __restrict__ row_idx, int n_sel, int agg,
                      const int32_t* __restrict__ seq_len, int64_t T_cap,
                      const int32_t* __restrict__ cand_pos, const int32_t* __restrict__ cand_count,
                      int C_cap, float* __restrict__ scores, int32_t* __restrict__ best_pos,
                      float* __restrict__ best_score, uint32_t* __restrict__ status) {
    extern __shared__ __align__(128) unsigned char dyn_smem[];
    int64_t* rows_sh = reinterpret_cast<int64_t*>(dyn_smem);   // element offset of each row
    __shared__ ArgmaxShared sh;
    __shared__ int bad_rows;

    cg::cluster_group cluster = cg::this_cluster();
    const int CL = static_cast<int>(cluster.num_blocks());
    const int rank = static_cast<int>(cluster.block_rank());
    const int b = blockIdx.x / CL;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    const int64_t L = seq_len[b];
    if (L < 0 || L > T_cap) {
        if (rank == 0 && tid == 0) {
            best_pos[b] = -1;
            if (best_score) best_score[b] = -INFINITY;
            if (status) status[b] |= PLDP_ST_SEQ_LEN;
        }
        return;
    }
    const int64_t t = L - 1;
    int n = cand_count[b];
    n = n < 0 ? 0 : (n > C_cap ? C_cap : n);
    const int stride_cand = CL * kWarps;
    const bool cta_work = rank < n;     // t < 1: listed candidates still get -inf scores
    const T* ab = A + static_cast<int64_t>(b) * seq_stride;

    if (tid == 0) bad_rows = 0;
    if (lane == 0) {
        sh.warp_key[warp] = 0;
        sh.warp_err[warp] = 0;
    }
    __syncthreads();
    for (int k = tid; k < n_sel; k += kThreads) {
        const int r = row_idx ? row_idx[k] : k;
        const bool okr = (r >= 0 && r < R);
        rows_sh[k] = okr ? static_cast<int64_t>(r) * row_stride : -1;
        if (!okr) bad_rows = 1;
    }
    __syncthreads();
    if (rank == 0 && tid == 0 && bad_rows && status) atomicOr(status + b, PLDP_ST_ROW_INDEX);

    if (cta_work) {
        constexpr int U = 4;
        for (int i = rank + CL * warp; i < n; i += stride_cand) {
            const int64_t j = cand_pos[static_cast<int64_t>(b) * C_cap + i];
            const bool ok = (j >= 0 && j < t);
            float s = -INFINITY;
            if (ok) {
                float acc = (agg == PLDP_AGG_MAX) ? -INFINITY : 0.0f;
                for (int k0 = lane; k0 < n_sel; k0 += 32 * U) {
                    float v[U];
#pragma unroll
                    for (int u = 0; u < U; ++u) {
                        const int k = k0 + 32 * u;
                        const int64_t off = (k < n_sel) ? rows_sh[k] : -1;
                        v[u] = (off >= 0) ? to_f32(ab[off + j]) : NAN;
                    }
#pragma unroll
                    for (int u = 0; u < U; ++u) {
                        if (v[u] == v[u]) acc = (agg == PLDP_AGG_MAX) ? fmaxf(acc, v[u]) : acc + v[u];
                    }
                }
                if (agg == PLDP_AGG_MAX) {
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) acc = fmaxf(acc, __shfl_xor_sync(0xFFFFFFFFu, acc, o));
                } else {
                    acc = warp_sum(acc);
                }
                s = acc;
            }
            if (lane == 0) {
                if (scores) scores[static_cast<int64_t>(b) * C_cap + i] = s;
                if (ok) {
                    const unsigned long long k = pack_key(s, static_cast<uint32_t>(j));
                    if (k > sh.warp_key[warp]) sh.warp_key[warp] = k;
                }
            }
        }
    }
    cluster_argmax_store(cluster, sh, b, best_pos, best_score, status, PLDP_ST_TIMEOUT);
}

int pick_cluster(int C_cap) {
    int cl = (C_cap + 2 * kWarps - 1) / (2 * kWarps);
    return cl < 1 ? 1 : (cl > kMaxCluster ? kMaxCluster : cl);
}

template <typename K, typename... Args>
cudaError_t launch_cluster(K kernel, int B, int CL, size_t smem, void* stream, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(B) * CL);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = static_cast<cudaStream_t>(stream);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CL;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

}  // namespace
}  // namespace pldp

using namespace pldp;

extern "C" PLDP_API pldp_status pldp_rank_hidden(const void* H, pldp_dtype dtype, int64_t d,
                                                 int64_t seq_stride, const int32_t* seq_len, int B,
                                                 int64_t T_cap, const int32_t* cand_pos,
                                                 const int32_t* cand_count, int C_cap,
                                                 float threshold, float* scores, int32_t* best_pos,
                                                 float* best_score, uint32_t* status, void* stream) {
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden: B < 0");
    if (dtype != PLDP_F32 && dtype != PLDP_BF16)
        return fail(PLDP_ERR_UNSUPPORTED, "rank_hidden: unsupported dtype %d", (int)dtype);
    const size_t es = dtype == PLDP_F32 ? 4 : 2;
    if (d < 1) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden: d < 1");
    if (static_cast<size_t>(d) * es > kMaxQueryBytes)
        return fail(PLDP_ERR_UNSUPPORTED, "rank_hidden: d * sizeof(dtype) > %zu", kMaxQueryBytes);
    if (T_cap < 0 || T_cap > INT32_MAX) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden: bad T_cap");
    if (seq_stride < T_cap * d) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden: seq_stride < T_cap*d");
    if (C_cap < 0) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden: C_cap < 0");
    if (threshold != threshold) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden: threshold is NaN");
    if (B == 0) return PLDP_OK;
    if (!H || !seq_len || !cand_count || !best_pos || (C_cap > 0 && !cand_pos))
        return fail(PLDP_ERR_INVALID_ARG, "rank_hidden: null pointer");

    const bool vec = aligned16(H) && (d * es) % 16 == 0 && (seq_stride * es) % 16 == 0;
    const int CL = pick_cluster(C_cap);
    const size_t smem = (static_cast<size_t>(d) * es + 127) / 128 * 128;
    cudaError_t e;
    if (dtype == PLDP_BF16) {
        const __nv_bfloat16* h = static_cast<const __nv_bfloat16*>(H);
        e = vec ? launch_cluster(rank_hidden_kernel<__nv_bfloat16, true>, B, CL, smem, stream, h, d,
                                 seq_stride, seq_len, T_cap, cand_pos, cand_count, C_cap, threshold,
                                 scores, best_pos, best_score, status)
                : launch_cluster(rank_hidden_kernel<__nv_bfloat16, false>, B, CL, smem, stream, h, d,
                                 seq_stride, seq_len, T_cap, cand_pos, cand_count, C_cap, threshold,
                                 scores, best_pos, best_score, status);
    } else {
        const float* h = static_cast<const float*>(H);
        e = vec ? launch_cluster(rank_hidden_kernel<float, true>, B, CL, smem, stream, h, d, seq_stride,
                                 seq_len, T_cap, cand_pos, cand_count, C_cap, threshold, scores,
                                 best_pos, best_score, status)
                : launch_cluster(rank_hidden_kernel<float, false>, B, CL, smem, stream, h, d,
                                 seq_stride, seq_len, T_cap, cand_pos, cand_count, C_cap, threshold,
                                 scores, best_pos, best_score, status);
    }
    if (e != cudaSuccess)
        return fail(PLDP_ERR_CUDA, "rank_hidden: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}

extern "C" PLDP_API pldp_status pldp_rank_attention(const void* A, pldp_dtype dtype, int R,
                                                    int64_t row_stride, int64_t seq_stride,
                                                    const int32_t* row_idx, int n_sel, pldp_agg agg,
                                                    const int32_t* seq_len, int B, int64_t T_cap,
                                                    const int32_t* cand_pos,
                                                    const int32_t* cand_count, int C_cap,
                                                    float* scores, int32_t* best_pos,
                                                    float* best_score, uint32_t* status,
                                                    void* stream) {
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "rank_attention: B < 0");
    if (dtype != PLDP_F32 && dtype != PLDP_BF16)
        return fail(PLDP_ERR_UNSUPPORTED, "rank_attention: unsupported dtype %d", (int)dtype);
    if (agg != PLDP_AGG_MAX && agg != PLDP_AGG_SUM)
        return fail(PLDP_ERR_INVALID_ARG, "rank_attention: unknown aggregation %d", (int)agg);
    if (R < 1) return fail(PLDP_ERR_INVALID_ARG, "rank_attention: R < 1");
    if (T_cap < 0 || T_cap > INT32_MAX) return fail(PLDP_ERR_INVALID_ARG, "rank_attention: bad T_cap");
    if (row_stride < T_cap) return fail(PLDP_ERR_INVALID_ARG, "rank_attention: row_stride < T_cap");
    if (seq_stride < static_cast<int64_t>(R) * row_stride)
        return fail(PLDP_ERR_INVALID_ARG, "rank_attention: seq_stride < R*row_stride");
    const int sel = row_idx ? n_sel : R;
    if (sel < 1 || sel > kMaxSelRows)
        return fail(PLDP_ERR_INVALID_ARG, "rank_attention: need 1 <= n_sel <= %d", kMaxSelRows);
    if (C_cap < 0) return fail(PLDP_ERR_INVALID_ARG, "rank_attention: C_cap < 0");
    if (B == 0) return PLDP_OK;
    if (!A || !seq_len || !cand_count || !best_pos || (C_cap > 0 && !cand_pos))
        return fail(PLDP_ERR_INVALID_ARG, "rank_attention: null pointer");

    const int CL = pick_cluster(C_cap);
    const size_t smem = static_cast<size_t>(sel) * sizeof(int64_t);
    cudaError_t e;
    if (dtype == PLDP_BF16)
        e = launch_cluster(rank_attention_kernel<__nv_bfloat16>, B, CL, smem, stream,
                           static_cast<const __nv_bfloat16*>(A), R, row_stride, seq_stride, row_idx,
                           sel, static_cast<int>(agg), seq_len, T_cap, cand_pos, cand_count, C_cap,
                           scores, best_pos, best_score, status);
    else
        e = launch_cluster(rank_attention_kernel<float>, B, CL, smem, stream,
                           static_cast<const float*>(A), R, row_stride, seq_stride, row_idx, sel,
                           static_cast<int>(agg), seq_len, T_cap, cand_pos, cand_count, C_cap, scores,
                           best_pos, best_score, status);
    if (e != cudaSuccess)
        return fail(PLDP_ERR_CUDA, "rank_attention: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}
