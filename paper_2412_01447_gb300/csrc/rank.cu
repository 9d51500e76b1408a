// Candidate ranking of PLD+:
//   hidden states -- Eq. 3 (Sec. 4.2.2): j* = argmax_{j in P} cos(H_{j-1}, H_{t-1})
//   attentions    -- Eq. 2 (Sec. 4.2.1): j* = argmax_{j in P} max_{(l,g) in L* x G*} A^{(l,g)}_{t-1}[j]
//
// Work layout.  S CTAs serve one sequence (S = 1 when the batch alone fills the
// GPU; for small batches S > 1 and the S CTAs form a thread-block cluster).
// Candidate i belongs to CTA i mod S.  A CTA scores its candidates P at a time
// (P = 1, 2, 4 or 8, the largest not above its count) with 8 / P warps per
// candidate, each warp taking an interleaved share of the row, so that a single
// candidate is read by the whole CTA in one round trip of DRAM latency while
// many candidates still stream with one warp each.  Partial sums meet in shared
// memory and are combined in a fixed order, so results are deterministic.
//
// The argmax uses packed (score, position) keys: the larger score wins, equal
// scores go to the smaller position, independent of reduction order.  With a
// cluster, CTA 0 combines the CTAs' keys over distributed shared memory.
//
// Hidden ranking stages the query row H_{t-1} in shared memory with one bulk
// asynchronous copy (when rows are 16-byte aligned), issued before the warps
// stream their candidate rows, so the two DRAM round trips overlap.
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

struct RankShared {
    float part[kWarps][3];                 // per-warp partial sums of the current batch
    unsigned long long slot_key[kWarps];   // best key seen by each candidate slot
    unsigned long long cta_key;
    int32_t jpre[kWarps];                  // prefetched positions of the first batch
    int cta_err;
    int err;
};

// Candidates of this CTA, and the batch shape for that count.
struct Batch {
    int n_local, P, G, slot, sub;
};

__device__ __forceinline__ Batch batch_shape(int n, int S, int rank, int warp) {
    Batch bt;
    bt.n_local = (n > rank) ? (n - rank + S - 1) / S : 0;
    bt.P = bt.n_local >= 8 ? 8 : (bt.n_local >= 4 ? 4 : (bt.n_local >= 2 ? 2 : 1));
    bt.G = kWarps / bt.P;
    bt.slot = warp / bt.G;
    bt.sub = warp - bt.slot * bt.G;
    return bt;
}

// Writes the best of this CTA (or of the cluster) for sequence b.  Reached by
// every thread of every CTA of the cluster.
template <bool CLUSTER>
__device__ __forceinline__ void store_best(RankShared& sh, int b, int32_t* best_pos,
                                           float* best_score, uint32_t* status, uint32_t err_bit) {
    const int tid = threadIdx.x;
    __syncthreads();
    if (tid == 0) {
        unsigned long long k = 0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) k = sh.slot_key[w] > k ? sh.slot_key[w] : k;
        sh.cta_key = k;
        sh.cta_err = sh.err;
    }
    unsigned long long k = 0;
    int err = 0;
    bool writer = false;
    if constexpr (CLUSTER) {
        cg::cluster_group cluster = cg::this_cluster();
        cluster.sync();
        if (cluster.block_rank() == 0 && tid < 32) {
            const int S = static_cast<int>(cluster.num_blocks());
            if (tid < S) {
                RankShared* remote = cluster.map_shared_rank(&sh, tid);
                k = remote->cta_key;
                err = remote->cta_err;
            }
            k = warp_max_u64(k);
            err = static_cast<int>(__reduce_or_sync(0xFFFFFFFFu, static_cast<unsigned>(err)));
            writer = (tid == 0);
        }
    } else {
        __syncthreads();
        if (tid == 0) {
            k = sh.cta_key;
            err = sh.cta_err;
            writer = true;
        }
    }
    if (writer) {
        if (err || k == 0) {
            best_pos[b] = -1;
            if (best_score) best_score[b] = -INFINITY;
            if (err && status) atomicOr(status + b, err_bit);
        } else {
            best_pos[b] = static_cast<int32_t>(key_index(k));
            if (best_score) best_score[b] = key_value(k);
        }
    }
    if constexpr (CLUSTER) {
        cl_arrive();
        cl_wait();   // CTA 0 has read every CTA's shared memory before any exits
    }
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

template <typename T, bool VEC, bool CLUSTER>
__global__ void __launch_bounds__(kThreads)
rank_hidden_kernel(const T* __restrict__ H, int64_t d, int64_t seq_stride,
                   const int32_t* __restrict__ seq_len, int64_t T_cap,
                   const int32_t* __restrict__ cand_pos, const int32_t* __restrict__ cand_count,
                   int C_cap, float threshold, float* __restrict__ scores,
                   int32_t* __restrict__ best_pos, float* __restrict__ best_score,
                   uint32_t* __restrict__ status, int S) {
    extern __shared__ __align__(128) unsigned char dyn_smem[];
    T* q_sh = reinterpret_cast<T*>(dyn_smem);          // query row H_{t-1}
    __shared__ RankShared sh;
    __shared__ __align__(8) uint64_t bar;

    const int b = blockIdx.x / S;
    const int rank = blockIdx.x - b * S;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    // The first candidate of every slot is fetched together with seq_len and the
    // count, saving a dependent round trip for the common small counts.
    if (lane == 0) {
        const int i_pre = rank + S * warp;
        sh.jpre[warp] = (i_pre < C_cap) ? cand_pos[static_cast<int64_t>(b) * C_cap + i_pre] : -1;
    }
    const int64_t L = seq_len[b];
    int n = cand_count[b];
    if (L < 0 || L > T_cap) {       // the same for every CTA of the sequence
        if (rank == 0 && tid == 0) {
            best_pos[b] = -1;
            if (best_score) best_score[b] = -INFINITY;
            if (status) atomicOr(status + b, PLDP_ST_SEQ_LEN);
        }
        return;
    }
    const int64_t t = L - 1;
    n = n < 0 ? 0 : (n > C_cap ? C_cap : n);
    const Batch bt = batch_shape(n, S, rank, warp);
    // With t < 2 no candidate is eligible (j >= 1 and j < t), but the listed
    // ones still get their -inf scores written.
    const bool need_query = bt.n_local > 0 && t >= 2;
    const T* hb = H + static_cast<int64_t>(b) * seq_stride;

    if (tid < kWarps) sh.slot_key[tid] = 0;
    if (tid == 0) sh.err = 0;
    bool q_ready = true;
    if (need_query) {
        const T* qg = hb + (t - 1) * d;
        if constexpr (VEC) {
            if (tid == 0) {
                mbar_init(&bar, 1);
                fence_mbar_init();
            }
            __syncthreads();
            if (tid == 0) {
                const uint32_t qbytes = static_cast<uint32_t>(d * sizeof(T));
                mbar_arrive_expect_tx(&bar, qbytes);
                bulk_g2s(q_sh, qg, qbytes, &bar);
            }
            q_ready = false;      // waited for right before the first use
        } else {
            for (int64_t k = tid; k < d; k += kThreads) q_sh[k] = qg[k];
        }
    }
    __syncthreads();

    bool timed_out = false;
    for (int k0 = 0; k0 < bt.n_local; k0 += bt.P) {
        const int k = k0 + bt.slot;
        const bool active = k < bt.n_local;
        const int i = rank + S * k;
        int64_t j = -1;
        if (active) j = (k0 == 0) ? sh.jpre[k] : cand_pos[static_cast<int64_t>(b) * C_cap + i];
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
                        if (!mbar_wait(&bar, 0, kMbarPolls)) timed_out = true;
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
        __syncthreads();
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
            if (scores) scores[static_cast<int64_t>(b) * C_cap + i] = s;
            if (ok && s > threshold) {
                const unsigned long long key = pack_key(s, static_cast<uint32_t>(j));
                if (key > sh.slot_key[bt.slot]) sh.slot_key[bt.slot] = key;
            }
        }
        __syncthreads();
        if (sh.err) break;                                // CTA-uniform after the barrier
    }
    if constexpr (VEC) {
        // The copy into this CTA's shared memory must have landed before exit (bounded).
        if (need_query && tid == 0 && !mbar_wait(&bar, 0, kMbarPolls)) sh.err = 1;
    }
    store_best<CLUSTER>(sh, b, best_pos, best_score, status, PLDP_ST_TIMEOUT);
}

// ---------------------------------------------------------------------------
// attention ranking
// ---------------------------------------------------------------------------
template <typename T, bool CLUSTER>
__global__ void __launch_bounds__(kThreads)
rank_attention_kernel(const T* __restrict__ A, int R, int64_t row_stride, int64_t seq_stride,
                      const int32_t* __restrict__ row_idx, int n_sel, int agg,
                      const int32_t* __restrict__ seq_len, int64_t T_cap,
                      const int32_t* __restrict__ cand_pos, const int32_t* __restrict__ cand_count,
                      int C_cap, float* __restrict__ scores, int32_t* __restrict__ best_pos,
                      float* __restrict__ best_score, uint32_t* __restrict__ status, int S) {
    extern __shared__ __align__(128) unsigned char dyn_smem[];
    int64_t* rows_sh = reinterpret_cast<int64_t*>(dyn_smem);   // element offset of each row
    __shared__ RankShared sh;
    __shared__ int bad_rows;

    const int b = blockIdx.x / S;
    const int rank = blockIdx.x - b * S;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    if (lane == 0) {
        const int i_pre = rank + S * warp;
        sh.jpre[warp] = (i_pre < C_cap) ? cand_pos[static_cast<int64_t>(b) * C_cap + i_pre] : -1;
    }
    const int64_t L = seq_len[b];
    int n = cand_count[b];
    if (L < 0 || L > T_cap) {
        if (rank == 0 && tid == 0) {
            best_pos[b] = -1;
            if (best_score) best_score[b] = -INFINITY;
            if (status) atomicOr(status + b, PLDP_ST_SEQ_LEN);
        }
        return;
    }
    const int64_t t = L - 1;
    n = n < 0 ? 0 : (n > C_cap ? C_cap : n);
    const Batch bt = batch_shape(n, S, rank, warp);
    const T* ab = A + static_cast<int64_t>(b) * seq_stride;

    if (tid == 0) {
        bad_rows = 0;
        sh.err = 0;
    }
    if (tid < kWarps) sh.slot_key[tid] = 0;
    __syncthreads();
    if (bt.n_local > 0 || rank == 0) {
        for (int k = tid; k < n_sel; k += kThreads) {
            const int r = row_idx ? row_idx[k] : k;
            const bool okr = (r >= 0 && r < R);
            rows_sh[k] = okr ? static_cast<int64_t>(r) * row_stride : -1;
            if (!okr) bad_rows = 1;
        }
    }
    __syncthreads();
    if (rank == 0 && tid == 0 && bad_rows && status) atomicOr(status + b, PLDP_ST_ROW_INDEX);

    const bool is_max = (agg == PLDP_AGG_MAX);
    constexpr int U = 4;
    for (int k0 = 0; k0 < bt.n_local; k0 += bt.P) {
        const int k = k0 + bt.slot;
        const bool active = k < bt.n_local;
        const int i = rank + S * k;
        int64_t j = -1;
        if (active) j = (k0 == 0) ? sh.jpre[k] : cand_pos[static_cast<int64_t>(b) * C_cap + i];
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
                    v[u] = (off >= 0) ? to_f32(ab[off + j]) : NAN;
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
        __syncthreads();
        if (bt.sub == 0 && lane == 0 && active) {
            float s = -INFINITY;
            if (ok) {
                s = sh.part[warp][0];
                for (int g = 1; g < bt.G; ++g)          // fixed order
                    s = is_max ? fmaxf(s, sh.part[warp + g][0]) : s + sh.part[warp + g][0];
            }
            if (scores) scores[static_cast<int64_t>(b) * C_cap + i] = s;
            if (ok) {
                const unsigned long long key = pack_key(s, static_cast<uint32_t>(j));
                if (key > sh.slot_key[bt.slot]) sh.slot_key[bt.slot] = key;
            }
        }
        __syncthreads();
    }
    store_best<CLUSTER>(sh, b, best_pos, best_score, status, PLDP_ST_TIMEOUT);
}

// CTAs per sequence: 1 when the batch fills the GPU, else up to a cluster of 8
// (never more than the candidate capacity).
int pick_split(int B, int C_cap) {
    int s = sm_count() / (B > 0 ? B : 1);
    if (s > C_cap) s = C_cap;
    return s < 1 ? 1 : (s > kMaxCluster ? kMaxCluster : s);
}

template <typename K, typename... Args>
cudaError_t launch_rank(K kernel, int B, int S, size_t smem, void* stream, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(B) * S);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = static_cast<cudaStream_t>(stream);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = S > 1 ? 1 : 0;
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    return cudaLaunchKernelEx(&cfg, kernel, args..., S);
}

template <typename T, bool VEC>
cudaError_t launch_hidden(int B, int S, size_t smem, void* stream, const T* h, int64_t d,
                          int64_t seq_stride, const int32_t* seq_len, int64_t T_cap,
                          const int32_t* cand_pos, const int32_t* cand_count, int C_cap,
                          float threshold, float* scores, int32_t* best_pos, float* best_score,
                          uint32_t* status) {
    if (S > 1)
        return launch_rank(rank_hidden_kernel<T, VEC, true>, B, S, smem, stream, h, d, seq_stride,
                           seq_len, T_cap, cand_pos, cand_count, C_cap, threshold, scores, best_pos,
                           best_score, status);
    return launch_rank(rank_hidden_kernel<T, VEC, false>, B, S, smem, stream, h, d, seq_stride,
                       seq_len, T_cap, cand_pos, cand_count, C_cap, threshold, scores, best_pos,
                       best_score, status);
}

template <typename T>
cudaError_t launch_attention(int B, int S, size_t smem, void* stream, const T* a, int R,
                             int64_t row_stride, int64_t seq_stride, const int32_t* row_idx, int sel,
                             int agg, const int32_t* seq_len, int64_t T_cap, const int32_t* cand_pos,
                             const int32_t* cand_count, int C_cap, float* scores, int32_t* best_pos,
                             float* best_score, uint32_t* status) {
    if (S > 1)
        return launch_rank(rank_attention_kernel<T, true>, B, S, smem, stream, a, R, row_stride,
                           seq_stride, row_idx, sel, agg, seq_len, T_cap, cand_pos, cand_count, C_cap,
                           scores, best_pos, best_score, status);
    return launch_rank(rank_attention_kernel<T, false>, B, S, smem, stream, a, R, row_stride,
                       seq_stride, row_idx, sel, agg, seq_len, T_cap, cand_pos, cand_count, C_cap,
                       scores, best_pos, best_score, status);
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
    const int S = pick_split(B, C_cap);
    const size_t smem = (static_cast<size_t>(d) * es + 127) / 128 * 128;
    cudaError_t e;
    if (dtype == PLDP_BF16) {
        const __nv_bfloat16* h = static_cast<const __nv_bfloat16*>(H);
        e = vec ? launch_hidden<__nv_bfloat16, true>(B, S, smem, stream, h, d, seq_stride, seq_len, T_cap,
                                                     cand_pos, cand_count, C_cap, threshold, scores,
                                                     best_pos, best_score, status)
                : launch_hidden<__nv_bfloat16, false>(B, S, smem, stream, h, d, seq_stride, seq_len,
                                                      T_cap, cand_pos, cand_count, C_cap, threshold,
                                                      scores, best_pos, best_score, status);
    } else {
        const float* h = static_cast<const float*>(H);
        e = vec ? launch_hidden<float, true>(B, S, smem, stream, h, d, seq_stride, seq_len, T_cap,
                                             cand_pos, cand_count, C_cap, threshold, scores, best_pos,
                                             best_score, status)
                : launch_hidden<float, false>(B, S, smem, stream, h, d, seq_stride, seq_len, T_cap,
                                              cand_pos, cand_count, C_cap, threshold, scores, best_pos,
                                              best_score, status);
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

    const int S = pick_split(B, C_cap);
    const size_t smem = static_cast<size_t>(sel) * sizeof(int64_t);
    cudaError_t e;
    if (dtype == PLDP_BF16)
        e = launch_attention<__nv_bfloat16>(B, S, smem, stream, static_cast<const __nv_bfloat16*>(A), R,
                                            row_stride, seq_stride, row_idx, sel, static_cast<int>(agg),
                                            seq_len, T_cap, cand_pos, cand_count, C_cap, scores,
                                            best_pos, best_score, status);
    else
        e = launch_attention<float>(B, S, smem, stream, static_cast<const float*>(A), R, row_stride,
                                    seq_stride, row_idx, sel, static_cast<int>(agg), seq_len, T_cap,
                                    cand_pos, cand_count, C_cap, scores, best_pos, best_score, status);
    if (e != cudaSuccess)
        return fail(PLDP_ERR_CUDA, "rank_attention: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}
