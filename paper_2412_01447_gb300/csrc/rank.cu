// pldp_rank_hidden (Eq. 3, Sec. 4.2.2) and pldp_rank_attention (Eq. 2, Sec. 4.2.1)
// as their own kernels, on the ranking blocks of pldp_rank.cuh.
//
// S CTAs serve one sequence: S = 1 when the batch alone fills the GPU; for small
// batches S > 1 and the S CTAs form a thread-block cluster whose CTA 0 combines
// their best keys over distributed shared memory.  Hidden ranking stages the
// query row H_{t-1} in shared memory with one bulk asynchronous copy (when rows
// are 16-byte aligned), issued before the warps stream their candidate rows, so
// the two DRAM round trips overlap.
#include <type_traits>

#include "pldp_rank.cuh"

namespace pldp {
namespace {

constexpr int kThreads = kRankThreads;
constexpr int kMaxCluster = 8;
constexpr size_t kMaxQueryBytes = 196608;     // d * sizeof(dtype) limit
constexpr int kMaxSelRows = 8192;             // row_idx entries staged in shared memory

struct CtaBest {
    unsigned long long key;
    int err;
};

// Writes the best of this CTA (or of the cluster) for sequence b.  Reached by
// every thread of every CTA of the cluster.
template <bool CLUSTER>
__device__ __forceinline__ void store_best(RankShared& sh, CtaBest& mine, int b, int32_t* best_pos,
                                           float* best_score, uint32_t* status, uint32_t err_bit) {
    const int tid = threadIdx.x;
    __syncthreads();
    if (tid == 0) {
        mine.key = rank_best_key(sh);
        mine.err = sh.err;
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
                CtaBest* remote = cluster.map_shared_rank(&mine, tid);
                k = remote->key;
                err = remote->err;
            }
            k = warp_max_u64(k);
            err = static_cast<int>(__reduce_or_sync(0xFFFFFFFFu, static_cast<unsigned>(err)));
            writer = (tid == 0);
        }
    } else {
        __syncthreads();
        if (tid == 0) {
            k = mine.key;
            err = mine.err;
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
        asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
        asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
    }
}

__device__ __forceinline__ void prefetch_first(RankShared& sh, const int32_t* cand_pos, int b, int C_cap,
                                               int S, int rank) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) {
        const int i = rank + S * warp;
        sh.jpre[warp] = (i < C_cap) ? cand_pos[static_cast<int64_t>(b) * C_cap + i] : -1;
    }
}

// 72 registers: the compiler's own choice for 256 threads was 64 with spills of the
// per-warp candidate stream (8 loads in flight per lane); without them, at 3 CTAs per
// SM, Eq. 3 on 510 candidates per sequence measured 116.6 -> 109.5 us (128 candidates:
// 42.8 -> 43.3 us), alternated on one box.
template <typename T, bool VEC, bool CLUSTER>
__global__ void __maxnreg__(72)
rank_hidden_kernel(const T* __restrict__ H, int64_t d, int64_t seq_stride,
                   const int32_t* __restrict__ seq_len, int64_t T_cap,
                   const int32_t* __restrict__ cand_pos, const int32_t* __restrict__ cand_count,
                   int C_cap, float threshold, float* __restrict__ scores,
                   int32_t* __restrict__ best_pos, float* __restrict__ best_score,
                   uint32_t* __restrict__ status, int S) {
    extern __shared__ __align__(128) unsigned char dyn_smem[];
    T* q_sh = reinterpret_cast<T*>(dyn_smem);          // query row H_{t-1}
    __shared__ RankShared sh;
    __shared__ CtaBest mine;
    __shared__ __align__(8) uint64_t bar;
#ifdef PLDP_TEST_STUCK_QUERY_WAIT
    // Test build only: the scoring warps wait for the query on a barrier that
    // nothing arrives on, so that their bounded wait runs out (the TIMEOUT path);
    // the copy itself still completes on `bar`, which is waited for before exit.
    __shared__ __align__(8) uint64_t stuck;
    uint64_t* const wait_bar = &stuck;
#else
    uint64_t* const wait_bar = &bar;
#endif

    pdl_enter();
    const int b = blockIdx.x / S;
    const int rank = blockIdx.x - b * S;
    const int tid = threadIdx.x;
    prefetch_first(sh, cand_pos, b, C_cap, S, rank);   // overlaps the seq_len/count loads
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
    // With t < 2 no candidate is eligible (j >= 1 and j < t), but the listed
    // ones still get their -inf scores written.
    const bool need_query = (n > rank) && t >= 2;
    const T* hb = H + static_cast<int64_t>(b) * seq_stride;
    rank_shared_init(sh);
    if (need_query) {
        const T* qg = hb + (t - 1) * d;
        if constexpr (VEC) {
            if (tid == 0) {
                mbar_init(&bar, 1);
                if (wait_bar != &bar) mbar_init(wait_bar, 1);
                fence_mbar_init();
                mbar_arrive_expect_tx(&bar, static_cast<uint32_t>(d * sizeof(T)));
                bulk_g2s(q_sh, qg, static_cast<uint32_t>(d * sizeof(T)), &bar);
            }
        } else {
            for (int64_t k = tid; k < d; k += kThreads) q_sh[k] = qg[k];
        }
    }
    __syncthreads();               // mbarrier initialised; shared state visible
    hidden_rank_cta<T, VEC>(hb, d, t, cand_pos + static_cast<int64_t>(b) * C_cap, n, S, rank, sh.jpre,
                            q_sh, wait_bar, need_query && VEC, threshold,
                            scores ? scores + static_cast<int64_t>(b) * C_cap : nullptr, sh);
    if constexpr (VEC) {
        // The copy into this CTA's shared memory must have landed before exit (bounded).
        if (need_query && tid == 0 && !mbar_wait(&bar, 0, kMbarPolls)) sh.err = 1;
    }
    store_best<CLUSTER>(sh, mine, b, best_pos, best_score, status, PLDP_ST_TIMEOUT);
}

// ---------------------------------------------------------------------------
// Averaged hidden states, the variant of Eq. 3 studied in App. B.2: every vector
// is replaced by the mean of the m rows ending at its position (cut at position
// 0), and candidate j scores cos(Hbar_{j-1}, Hbar_{t-1}).  Window sums are used
// in place of means (the cosine ignores the positive factor).  The query's
// window sum is built once in shared memory in fp32; each candidate's is formed
// on the fly by the whole CTA -- thread i takes chunks i, i + 256, ... -- and the
// partial sums meet in warp order.  One candidate at a time per CTA.
// ---------------------------------------------------------------------------
constexpr size_t kMaxAvgQueryBytes = 196608;   // d * 4: the fp32 window sum of the query

template <typename T, bool VEC>
struct Chunk {
    static constexpr int E = VEC ? 16 / static_cast<int>(sizeof(T)) : 1;
    using Raw = typename std::conditional<VEC, uint4, T>::type;
    static __device__ __forceinline__ Raw load(const T* p) {
        if constexpr (VEC) return ld_stream16(p);
        else return *p;
    }
    // Adds the E elements of x to acc.
    static __device__ __forceinline__ void add(const Raw& x, float (&acc)[E]) {
        if constexpr (VEC) {
            const uint32_t w[4] = {x.x, x.y, x.z, x.w};
            if constexpr (sizeof(T) == 2) {
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    acc[2 * k] += __uint_as_float(w[k] << 16);
                    acc[2 * k + 1] += __uint_as_float(w[k] & 0xFFFF0000u);
                }
            } else {
#pragma unroll
                for (int k = 0; k < 4; ++k) acc[k] += __uint_as_float(w[k]);
            }
        } else {
            acc[0] += to_f32(x);
        }
    }
    // acc = sum of the chunks at p + r * d for rows r in [lo, hi], four loads in flight.
    static __device__ __forceinline__ void window(const T* p, int64_t d, int64_t lo, int64_t hi, float (&acc)[E]) {
#pragma unroll
        for (int e = 0; e < E; ++e) acc[e] = 0.f;
        for (int64_t r0 = lo; r0 <= hi; r0 += 4) {
            Raw x[4];
#pragma unroll
            for (int u = 0; u < 4; ++u)
                if (r0 + u <= hi) x[u] = load(p + (r0 + u) * d);
#pragma unroll
            for (int u = 0; u < 4; ++u)
                if (r0 + u <= hi) add(x[u], acc);
        }
    }
};

template <typename T, bool VEC, bool CLUSTER>
__global__ void __launch_bounds__(kThreads)
rank_hidden_avg_kernel(const T* __restrict__ H, int64_t d, int64_t seq_stride, int m,
                       const int32_t* __restrict__ seq_len, int64_t T_cap,
                       const int32_t* __restrict__ cand_pos, const int32_t* __restrict__ cand_count,
                       int C_cap, float threshold, float* __restrict__ scores,
                       int32_t* __restrict__ best_pos, float* __restrict__ best_score,
                       uint32_t* __restrict__ status, int S) {
    using C = Chunk<T, VEC>;
    constexpr int E = C::E;
    extern __shared__ __align__(128) unsigned char dyn_smem[];
    float* qs = reinterpret_cast<float*>(dyn_smem);       // window sum ending at H_{t-1}
    __shared__ RankShared sh;
    __shared__ CtaBest mine;

    pdl_enter();
    const int b = blockIdx.x / S;
    const int rank = blockIdx.x - b * S;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
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
    const T* hb = H + static_cast<int64_t>(b) * seq_stride;
    const int64_t nch = d / E;
    rank_shared_init(sh);
    if (n > rank && t >= 2) {
        const int64_t lo = t - m > 0 ? t - m : 0;                 // rows lo .. t-1
        for (int64_t c = tid; c < nch; c += kThreads) {
            float acc[E];
            C::window(hb + c * E, d, lo, t - 1, acc);
#pragma unroll
            for (int e = 0; e < E; ++e) qs[c * E + e] = acc[e];
        }
    }
    __syncthreads();
    const int32_t* cands = cand_pos + static_cast<int64_t>(b) * C_cap;
    for (int i = rank; i < n; i += S) {                           // CTA-uniform
        const int64_t j = __ldg(cands + i);
        const bool ok = j >= 1 && j < t;
        float dot = 0.f, na = 0.f, nq = 0.f;
        if (ok) {
            const int64_t lo = j - m > 0 ? j - m : 0;             // rows lo .. j-1
            for (int64_t c = tid; c < nch; c += kThreads) {
                float a[E];
                C::window(hb + c * E, d, lo, j - 1, a);
#pragma unroll
                for (int e = 0; e < E; ++e) {
                    const float q = qs[c * E + e];
                    dot = fmaf(a[e], q, dot);
                    na = fmaf(a[e], a[e], na);
                    nq = fmaf(q, q, nq);
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
        __syncthreads();
        if (tid == 0) {
            float s = -INFINITY;
            if (ok) {
                float D = 0.f, N = 0.f, Q = 0.f;
                for (int w = 0; w < kRankWarps; ++w) {            // fixed order
                    D += sh.part[w][0];
                    N += sh.part[w][1];
                    Q += sh.part[w][2];
                }
                s = finish_cosine(D, N, Q);
            }
            if (scores) scores[static_cast<int64_t>(b) * C_cap + i] = s;
            if (ok && s > threshold) {
                const unsigned long long key = pack_key(s, static_cast<uint32_t>(j));
                if (key > sh.slot_key[0]) sh.slot_key[0] = key;
            }
        }
        __syncthreads();
    }
    store_best<CLUSTER>(sh, mine, b, best_pos, best_score, status, PLDP_ST_TIMEOUT);
}

// DENSE: all R rows in order, each key's values one run of dense_nv 16-byte vectors
// (checked on the host), ranked under MAX with whole-vector loads.
template <bool CLUSTER, bool DENSE>
__global__ void __launch_bounds__(kThreads)
rank_attention_kernel(const void* __restrict__ A, bool a_bf16, int R, int64_t row_stride, int64_t key_stride,
                      int64_t seq_stride, const int32_t* __restrict__ row_idx, int n_sel, int agg, int dense_nv,
                      const int32_t* __restrict__ seq_len, int64_t T_cap,
                      const int32_t* __restrict__ cand_pos, const int32_t* __restrict__ cand_count,
                      int C_cap, float* __restrict__ scores, int32_t* __restrict__ best_pos,
                      float* __restrict__ best_score, uint32_t* __restrict__ status, int S) {
    extern __shared__ __align__(128) unsigned char dyn_smem[];
    int64_t* rows_sh = reinterpret_cast<int64_t*>(dyn_smem);   // element offset of each row
    __shared__ RankShared sh;
    __shared__ CtaBest mine;
    __shared__ int bad_rows;

    pdl_enter();
    const int b = blockIdx.x / S;
    const int rank = blockIdx.x - b * S;
    const int tid = threadIdx.x;
    prefetch_first(sh, cand_pos, b, C_cap, S, rank);
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
    rank_shared_init(sh);
    const bool bad = stage_rows(rows_sh, row_idx, n_sel, R, row_stride, &bad_rows);
    if (rank == 0 && tid == 0 && bad && status) atomicOr(status + b, PLDP_ST_ROW_INDEX);
    const size_t es = a_bf16 ? 2 : 4;
    const void* ab = static_cast<const char*>(A) + static_cast<int64_t>(b) * seq_stride * es;
    attention_rank_cta(ab, a_bf16, rows_sh, n_sel, key_stride, t, cand_pos + static_cast<int64_t>(b) * C_cap, n, S,
                       rank, sh.jpre, agg == PLDP_AGG_MAX,
                       scores ? scores + static_cast<int64_t>(b) * C_cap : nullptr, sh, whole_cta(),
                       DENSE ? dense_nv : 0);
    store_best<CLUSTER>(sh, mine, b, best_pos, best_score, status, PLDP_ST_TIMEOUT);
}

// CTAs per sequence: as many as the kernel's resident CTA slots allow for the
// batch (all of its CTAs in one wave), up to a cluster of 8, never more than the
// candidate capacity.  `kernel` is the variant launched when S > 1.
int pick_split(int B, int C_cap, const void* kernel, size_t smem) {
    int s = resident_blocks(kernel, kThreads, smem) / (B > 0 ? B : 1);
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
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = S;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = S > 1 ? 2 : 1;
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

template <bool DENSE>
cudaError_t launch_attention(int B, int S, size_t smem, void* stream, const void* a, bool a_bf16,
                             int R, int64_t row_stride, int64_t key_stride, int64_t seq_stride, const int32_t* row_idx,
                             int sel, int agg, int dense_nv, const int32_t* seq_len, int64_t T_cap,
                             const int32_t* cand_pos, const int32_t* cand_count, int C_cap,
                             float* scores, int32_t* best_pos, float* best_score, uint32_t* status) {
    if (S > 1)
        return launch_rank(rank_attention_kernel<true, DENSE>, B, S, smem, stream, a, a_bf16, R, row_stride,
                           key_stride, seq_stride, row_idx, sel, agg, dense_nv, seq_len, T_cap, cand_pos, cand_count,
                           C_cap, scores, best_pos, best_score, status);
    return launch_rank(rank_attention_kernel<false, DENSE>, B, S, smem, stream, a, a_bf16, R, row_stride, key_stride,
                       seq_stride, row_idx, sel, agg, dense_nv, seq_len, T_cap, cand_pos, cand_count, C_cap,
                       scores, best_pos, best_score, status);
}

// Vectors per key of the dense form of Eq. 2 (all rows in order, row stride 1, every
// run 16-byte aligned, a power of two of vectors up to 32 * kDenseLoads), or 0.
int dense_vectors(const void* A, size_t es, int R, int64_t row_stride, int64_t key_stride, int64_t seq_stride,
                  const int32_t* row_idx, pldp_agg agg) {
    if (agg != PLDP_AGG_MAX || row_idx || row_stride != 1 || !aligned16(A)) return 0;
    if ((key_stride * static_cast<int64_t>(es)) % 16 || (seq_stride * static_cast<int64_t>(es)) % 16) return 0;
    const int64_t bytes = static_cast<int64_t>(R) * static_cast<int64_t>(es);
    if (bytes % 16) return 0;
    const int64_t nv = bytes / 16;
    if (nv > 32 * kDenseLoads || (nv & (nv - 1))) return 0;
    return static_cast<int>(nv);
}

template <typename T, bool VEC>
cudaError_t launch_hidden_avg(int B, int S, size_t smem, void* stream, const T* h, int64_t d, int64_t seq_stride,
                              int m, const int32_t* seq_len, int64_t T_cap, const int32_t* cand_pos,
                              const int32_t* cand_count, int C_cap, float threshold, float* scores,
                              int32_t* best_pos, float* best_score, uint32_t* status) {
    if (S > 1)
        return launch_rank(rank_hidden_avg_kernel<T, VEC, true>, B, S, smem, stream, h, d, seq_stride, m, seq_len,
                           T_cap, cand_pos, cand_count, C_cap, threshold, scores, best_pos, best_score, status);
    return launch_rank(rank_hidden_avg_kernel<T, VEC, false>, B, S, smem, stream, h, d, seq_stride, m, seq_len,
                       T_cap, cand_pos, cand_count, C_cap, threshold, scores, best_pos, best_score, status);
}

}  // namespace
}  // namespace pldp

using namespace pldp;

extern "C" PLDP_API pldp_status pldp_rank_hidden_avg(const void* H, pldp_dtype dtype, int64_t d,
                                                     int64_t seq_stride, int m, const int32_t* seq_len,
                                                     int B, int64_t T_cap, const int32_t* cand_pos,
                                                     const int32_t* cand_count, int C_cap, float threshold,
                                                     float* scores, int32_t* best_pos, float* best_score,
                                                     uint32_t* status, void* stream) {
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden_avg: B < 0");
    if (dtype != PLDP_F32 && dtype != PLDP_BF16)
        return fail(PLDP_ERR_UNSUPPORTED, "rank_hidden_avg: unsupported dtype %d", (int)dtype);
    const size_t es = dtype == PLDP_F32 ? 4 : 2;
    if (d < 1) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden_avg: d < 1");
    if (m < 1) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden_avg: m < 1");
    if (static_cast<size_t>(d) * sizeof(float) > kMaxAvgQueryBytes)
        return fail(PLDP_ERR_UNSUPPORTED, "rank_hidden_avg: d * 4 > %zu", kMaxAvgQueryBytes);
    if (T_cap < 0 || T_cap > INT32_MAX) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden_avg: bad T_cap");
    if (seq_stride < T_cap * d) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden_avg: seq_stride < T_cap*d");
    if (C_cap < 0) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden_avg: C_cap < 0");
    if (threshold != threshold) return fail(PLDP_ERR_INVALID_ARG, "rank_hidden_avg: threshold is NaN");
    if (B == 0) return PLDP_OK;
    if (!H || !seq_len || !cand_count || !best_pos || (C_cap > 0 && !cand_pos))
        return fail(PLDP_ERR_INVALID_ARG, "rank_hidden_avg: null pointer");

    const bool vec = aligned16(H) && (d * es) % 16 == 0 && (seq_stride * es) % 16 == 0;
    const size_t smem = (static_cast<size_t>(d) * sizeof(float) + 127) / 128 * 128;
    const int S = pick_split(B, C_cap, reinterpret_cast<const void*>(&rank_hidden_avg_kernel<__nv_bfloat16, true, true>),
                             smem);
    cudaError_t e;
    if (dtype == PLDP_BF16) {
        const __nv_bfloat16* h = static_cast<const __nv_bfloat16*>(H);
        e = vec ? launch_hidden_avg<__nv_bfloat16, true>(B, S, smem, stream, h, d, seq_stride, m, seq_len, T_cap,
                                                         cand_pos, cand_count, C_cap, threshold, scores, best_pos,
                                                         best_score, status)
                : launch_hidden_avg<__nv_bfloat16, false>(B, S, smem, stream, h, d, seq_stride, m, seq_len, T_cap,
                                                          cand_pos, cand_count, C_cap, threshold, scores, best_pos,
                                                          best_score, status);
    } else {
        const float* h = static_cast<const float*>(H);
        e = vec ? launch_hidden_avg<float, true>(B, S, smem, stream, h, d, seq_stride, m, seq_len, T_cap, cand_pos,
                                                 cand_count, C_cap, threshold, scores, best_pos, best_score, status)
                : launch_hidden_avg<float, false>(B, S, smem, stream, h, d, seq_stride, m, seq_len, T_cap, cand_pos,
                                                  cand_count, C_cap, threshold, scores, best_pos, best_score,
                                                  status);
    }
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "rank_hidden_avg: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}

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
    const size_t smem = (static_cast<size_t>(d) * es + 127) / 128 * 128;
    const int S = pick_split(B, C_cap, reinterpret_cast<const void*>(&rank_hidden_kernel<__nv_bfloat16, true, true>),
                             smem);
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
                                                    int64_t row_stride, int64_t key_stride, int64_t seq_stride,
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
    if (key_stride == 0) key_stride = 1;
    if (const char* why = attention_layout_error(R, T_cap, row_stride, key_stride, seq_stride))
        return fail(PLDP_ERR_INVALID_ARG, "rank_attention: %s", why);
    const int sel = row_idx ? n_sel : R;
    if (sel < 1 || sel > kMaxSelRows)
        return fail(PLDP_ERR_INVALID_ARG, "rank_attention: need 1 <= n_sel <= %d", kMaxSelRows);
    if (C_cap < 0) return fail(PLDP_ERR_INVALID_ARG, "rank_attention: C_cap < 0");
    if (B == 0) return PLDP_OK;
    if (!A || !seq_len || !cand_count || !best_pos || (C_cap > 0 && !cand_pos))
        return fail(PLDP_ERR_INVALID_ARG, "rank_attention: null pointer");

    const size_t smem = static_cast<size_t>(sel) * sizeof(int64_t);
    const int nv = dense_vectors(A, dtype == PLDP_F32 ? 4 : 2, R, row_stride, key_stride, seq_stride, row_idx, agg);
    cudaError_t e;
    if (nv > 0) {
        const int S = pick_split(B, C_cap, reinterpret_cast<const void*>(&rank_attention_kernel<true, true>), smem);
        e = launch_attention<true>(B, S, smem, stream, A, dtype == PLDP_BF16, R, row_stride, key_stride, seq_stride,
                                   row_idx, sel, static_cast<int>(agg), nv, seq_len, T_cap, cand_pos, cand_count, C_cap,
                                   scores, best_pos, best_score, status);
    } else {
        const int S = pick_split(B, C_cap, reinterpret_cast<const void*>(&rank_attention_kernel<true, false>), smem);
        e = launch_attention<false>(B, S, smem, stream, A, dtype == PLDP_BF16, R, row_stride, key_stride, seq_stride,
                                    row_idx, sel, static_cast<int>(agg), 0, seq_len, T_cap, cand_pos, cand_count,
                                    C_cap, scores, best_pos, best_score, status);
    }
    if (e != cudaSuccess)
        return fail(PLDP_ERR_CUDA, "rank_attention: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}
