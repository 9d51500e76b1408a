// Draft prediction (Sec. 4.3) and greedy verification (Sec. 4.4) of PLD+.
//
// Verification is two kernels chained by programmatic dependent launch.
//
// 1. One streaming pass over the flattened logits [B, K+1, V], cut into 2 KB
//    segments.  Warp w of the W in the grid takes segments w, w + W, w + 2W, ...
//    so the segments in flight form a moving window over memory, and the grid
//    is several waves of small CTAs, so the block scheduler keeps every SM busy
//    to the end (faster SMs take more CTAs).  Each lane issues its four 16-byte
//    loads of a segment at once and keeps a running (max, first index) with a
//    packed max over each vector, so the index search runs only when the max
//    grows.  A segment crosses at most one row boundary (rows are longer than a
//    segment on this path); per row, the warps' results meet in a packed 64-bit
//    key (value, inverted index) combined with atomicMax in the workspace, which
//    makes the argmax exact and independent of scheduling: larger value wins,
//    the smaller index wins ties, -0.0 equals +0.0.  The pass never waits on
//    another warp and never fences.
// 2. One warp per sequence reads its K+1 row keys, finds the accepted length and
//    the bonus token, appends them to the context and returns the keys to zero
//    for the next call.  Its launch is hidden behind the pass's last wave.
#include <math.h>

#include "pldp_internal.cuh"
#include "pldp_verify.cuh"

namespace pldp {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 8;                  // loads in flight per lane on the row-loop path
constexpr int kSegLoads = 4;                // 16-byte loads per lane per segment
constexpr int64_t kSegBytes = 32 * kSegLoads * 16;   // 2 KB
constexpr int kPassBlocksPerSm = 8;         // register cap: 8 CTAs of 8 warps per SM
constexpr int kPassWaves = 6;               // grid = up to 6 waves of resident CTAs

__global__ void extract_draft_kernel(const int32_t* __restrict__ ids, int64_t ids_stride,
                                     const int32_t* __restrict__ seq_len, int64_t T_cap,
                                     const int32_t* __restrict__ best_pos, int B, int K,
                                     int32_t* __restrict__ draft, int32_t* __restrict__ draft_len) {
    pdl_enter();
    const int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= static_cast<int64_t>(B) * K) return;
    const int b = static_cast<int>(idx / K);
    const int i = static_cast<int>(idx - static_cast<int64_t>(b) * K);
    const int64_t L = seq_len[b];
    const int64_t js = best_pos[b];
    const int64_t t = L - 1;
    int64_t d = 0;
    if (L >= 0 && L <= T_cap && js >= 0 && js < t) d = (t - js < K) ? (t - js) : K;
    draft[idx] = (i < d) ? ids[static_cast<int64_t>(b) * ids_stride + js + 1 + i] : -1;
    if (i == 0) draft_len[b] = static_cast<int32_t>(d);
}

// Running (max, first index) of one lane over elements [c0, c1) of a row.
template <typename T, bool VEC>
__device__ __forceinline__ void lane_argmax(const T* __restrict__ row, int64_t c0, int64_t c1,
                                            int lane, float& bv, int64_t& bi) {
    if constexpr (VEC) {
        constexpr int VW = 16 / sizeof(T);
        const uint4* p = reinterpret_cast<const uint4*>(row);
        const int64_t v0 = c0 / VW, v1 = c1 / VW;
        for (int64_t vb = v0 + lane; vb < v1; vb += 32 * kUnroll) {
            uint4 x[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int64_t v = vb + 32 * u;
                if (v < v1) x[u] = ld_stream16(p + v);
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int64_t v = vb + 32 * u;
                if (v < v1) {
                    const float m = vmax(x[u], T());
                    if (m > bv) {
                        bv = m;
                        bi = v * VW + vfirst(x[u], m, T());
                    }
                }
            }
        }
    } else {
        for (int64_t cb = c0 + lane; cb < c1; cb += 32 * kUnroll) {
            float x[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int64_t c = cb + 32 * u;
                x[u] = (c < c1) ? to_f32(row[c]) : -INFINITY;
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                if (x[u] > bv) {
                    bv = x[u];
                    bi = cb + 32 * u;
                }
            }
        }
    }
}

// Packed key from an ordered value key (see ordered_key) and an index.
__device__ __forceinline__ unsigned long long pack_ordered(uint32_t okey, uint32_t idx) {
    return (static_cast<unsigned long long>(okey) << 32) | static_cast<unsigned long long>(0xFFFFFFFFu - idx);
}

// Segment [s0, s0 + 32 * kSegLoads) of the flattened logits, in 16-byte vectors
// (nvec in all, vrow per row, rows at least a segment long, nvec < 2^31 so that
// 32-bit indices hold).  The segment starts `rem` vectors into row r0.
//
// Common case, the segment inside row r0: each lane takes the max of its four
// vectors, the warp's max comes from one redux over the ordered keys, and only
// the lane(s) holding it search for the element; a second redux picks the
// smallest index.  A segment that crosses into row r0 + 1 keeps a running
// (max, first index) per row and lane.
struct SegKeys {
    unsigned long long k0;   // the segment's best in its first row
    unsigned long long k1;   // ... in the next row when the segment crosses into it, else 0
};

template <typename T>
__device__ __forceinline__ SegKeys segment_argmax(const uint4* __restrict__ p, uint32_t s0, uint32_t nvec,
                                                  uint32_t r0, uint32_t rem, uint32_t vrow, int lane) {
    constexpr uint32_t VW = 16 / sizeof(T);
    constexpr uint32_t seg = 32 * kSegLoads;
    uint4 x[kSegLoads];
#pragma unroll
    for (int u = 0; u < kSegLoads; ++u) {
        const uint32_t v = s0 + lane + 32 * u;
        if (v < nvec) x[u] = ld_stream16(p + v);
    }
    if (rem + seg <= vrow && s0 + seg <= nvec) {               // warp-uniform
        float m = vmax(x[0], T());
#pragma unroll
        for (int u = 1; u < kSegLoads; ++u) m = fmaxf(m, vmax(x[u], T()));
        const uint32_t ok = ordered_key(m);
        const uint32_t wk = __reduce_max_sync(0xFFFFFFFFu, ok);
        uint32_t idx = 0xFFFFFFFFu;
        if (ok == wk) {
#pragma unroll
            for (int u = 0; u < kSegLoads; ++u)
                if (idx == 0xFFFFFFFFu && vmax(x[u], T()) == m)
                    idx = (rem + lane + 32 * u) * VW + vfirst(x[u], m, T());
        }
        idx = __reduce_min_sync(0xFFFFFFFFu, idx);
        return SegKeys{pack_ordered(wk, idx), 0ull};
    }
    const uint32_t bnd = s0 - rem + vrow;                      // first vector of row r0 + 1
    float b0 = -INFINITY, b1 = -INFINITY;
    uint32_t i0 = rem * VW, i1 = 0;
#pragma unroll
    for (int u = 0; u < kSegLoads; ++u) {
        const uint32_t v = s0 + lane + 32 * u;
        if (v < nvec) {
            const float m = vmax(x[u], T());
            if (v < bnd) {
                if (m > b0) {
                    b0 = m;
                    i0 = (v - (s0 - rem)) * VW + vfirst(x[u], m, T());
                }
            } else if (m > b1) {
                b1 = m;
                i1 = (v - bnd) * VW + vfirst(x[u], m, T());
            }
        }
    }
    const unsigned long long k0 = warp_max_u64(pack_key(b0, i0));
    unsigned long long k1 = 0ull;
    if (s0 + seg > bnd && bnd < nvec) k1 = warp_max_u64(pack_key(b1, i1));
    return SegKeys{k0, k1};
}

// Any segment: row by row, each row piece with the lane loop above.
template <typename T, bool VEC>
__device__ __forceinline__ void segment_rows(const T* __restrict__ logits, int64_t e0, int64_t e1, int64_t V,
                                             int lane, unsigned long long* __restrict__ keys) {
    for (int64_t pos = e0; pos < e1;) {
        const int64_t r = pos / V;
        const int64_t c0 = pos - r * V;
        const int64_t c1 = (V < c0 + (e1 - pos)) ? V : c0 + (e1 - pos);
        float bv = -INFINITY;
        int64_t bi = c0;
        lane_argmax<T, VEC>(logits + r * V, c0, c1, lane, bv, bi);
        const unsigned long long k = warp_max_u64(pack_key(bv, static_cast<uint32_t>(bi)));
        if (lane == 0) atomicMax(keys + r, k);
        pos += c1 - c0;
    }
}

// 1. the row argmax pass.  W = warps in the grid.  PATH 0: 16-byte loads, rows of
// at least a segment (the streaming path); 1: 16-byte loads, short rows; 2: element
// loads (unaligned logits or rows that are not a whole number of 16 bytes).
template <typename T, int PATH>
__global__ void __launch_bounds__(kThreads, PATH == 0 ? kPassBlocksPerSm : 4)
verify_argmax_kernel(const T* __restrict__ logits, int64_t N, int64_t V, int64_t W,
                     unsigned long long* __restrict__ keys) {
    pdl_enter();
    const int lane = threadIdx.x & 31;
    const int64_t w = static_cast<int64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
    if constexpr (PATH == 0) {
        // Per round the CTA's warps hold 8 consecutive segments (16 KB, rarely more
        // than one row): their keys meet in shared memory and thread 0 issues one
        // atomicMax per row touched.  Rounds are counted from the CTA's first warp,
        // so every warp takes part in every round (with no segment past the end).
        __shared__ unsigned long long sk[2][kWarps][2];
        __shared__ uint32_t srow[2][kWarps];
        const int warp = threadIdx.x >> 5;
        constexpr uint32_t VW = 16 / sizeof(T);
        constexpr uint32_t seg = 32 * kSegLoads;
        const uint32_t nvec = static_cast<uint32_t>(N / VW), vrow = static_cast<uint32_t>(V / VW);
        const uint32_t stride = static_cast<uint32_t>(W) * seg;
        const uint4* p = reinterpret_cast<const uint4*>(logits);
        const uint32_t dq = stride / vrow, dr = stride - dq * vrow;      // rows and vectors per stride
        uint32_t s0 = static_cast<uint32_t>(w) * seg;
        uint32_t r0 = s0 / vrow, rem = s0 - r0 * vrow;
        uint32_t first = blockIdx.x * kWarps * seg;                       // the CTA's first segment
        for (int buf = 0; first < nvec; first += stride, buf ^= 1) {
            const bool mine = s0 < nvec;
            SegKeys k = {0ull, 0ull};
            if (mine) k = segment_argmax<T>(p, s0, nvec, r0, rem, vrow, lane);
            if (lane == 0) {
                srow[buf][warp] = mine ? r0 : 0xFFFFFFFFu;
                sk[buf][warp][0] = k.k0;
                sk[buf][warp][1] = k.k1;
            }
            __syncthreads();
            if (threadIdx.x == 0) {                                       // rows are nondecreasing here
                uint32_t cur = 0xFFFFFFFFu;
                unsigned long long best = 0ull;
                for (int q = 0; q < kWarps; ++q) {
                    const uint32_t r = srow[buf][q];
                    if (r == 0xFFFFFFFFu) continue;
                    if (r != cur) {
                        if (cur != 0xFFFFFFFFu) atomicMax(keys + cur, best);
                        cur = r;
                        best = 0ull;
                    }
                    best = sk[buf][q][0] > best ? sk[buf][q][0] : best;
                    if (sk[buf][q][1]) {                                  // it crosses into row r + 1
                        atomicMax(keys + cur, best);
                        cur = r + 1;
                        best = sk[buf][q][1];
                    }
                }
                if (cur != 0xFFFFFFFFu) atomicMax(keys + cur, best);
            }
            s0 += stride;
            r0 += dq;
            rem += dr;
            if (rem >= vrow) {
                rem -= vrow;
                ++r0;
            }
        }
    } else {
        constexpr int64_t SEG = kSegBytes / static_cast<int64_t>(sizeof(T));   // elements per segment
        for (int64_t e0 = w * SEG; e0 < N; e0 += W * SEG) {
            const int64_t e1 = e0 + SEG < N ? e0 + SEG : N;
            segment_rows<T, PATH == 1>(logits, e0, e1, V, lane, keys);
        }
    }
}

// 2. accept, bonus and append: one warp per sequence.
__global__ void __launch_bounds__(kThreads) verify_finish_kernel(VerifyArgs a) {
    pdl_enter();                                           // the pass's keys are final
    const int64_t b = static_cast<int64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
    if (b < a.B) finish_sequence(a, b, threadIdx.x & 31, KeyTokens{a.row_keys + b * (a.K + 1)});
}

size_t keys_bytes(int B, int K) {
    return (static_cast<size_t>(B) * (K + 1) * sizeof(unsigned long long) + 255) / 256 * 256;
}

// Sizes the pass's grid (up to kPassWaves waves of resident CTAs, no more warps
// than segments) and launches it.  `a` has everything but the keys.
template <typename T, int PATH>
pldp_status launch_pass_t(const void* logits, VerifyArgs& a, void* scratch, cudaStream_t s, const char* what) {
    const void* fn = reinterpret_cast<const void*>(&verify_argmax_kernel<T, PATH>);
    const int64_t N = static_cast<int64_t>(a.B) * (a.K + 1) * a.V;
    constexpr int64_t SEG = kSegBytes / static_cast<int64_t>(sizeof(T));
    const int64_t segs = (N + SEG - 1) / SEG;
    int64_t blocks = static_cast<int64_t>(resident_blocks(fn, kThreads, 0)) * kPassWaves;
    const int64_t need = (segs + kWarps - 1) / kWarps;
    if (blocks > need) blocks = need;
    if (blocks < 1) blocks = 1;
    a.row_keys = static_cast<unsigned long long*>(scratch);
    const cudaError_t e = launch_pdl(verify_argmax_kernel<T, PATH>, dim3(static_cast<unsigned>(blocks)),
                                     dim3(kThreads), 0, s, 0, static_cast<const T*>(logits), N,
                                     static_cast<int64_t>(a.V), blocks * kWarps, a.row_keys);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "%s: launch failed: %s", what, cudaGetErrorString(e));
    return PLDP_OK;
}

}  // namespace

pldp_status launch_verify_pass(const void* logits, pldp_dtype dtype, VerifyArgs& a, void* scratch,
                               cudaStream_t s, const char* what) {
    const size_t es = dtype == PLDP_F32 ? 4 : 2;
    const bool vec = aligned16(logits) && (static_cast<size_t>(a.V) * es) % 16 == 0;
    const int64_t bytes = static_cast<int64_t>(a.B) * (a.K + 1) * a.V * static_cast<int64_t>(es);
    const bool long_rows = static_cast<int64_t>(a.V) * static_cast<int64_t>(es) >= kSegBytes;
    const bool small = bytes / 16 < (int64_t(1) << 31);     // 32-bit vector indices
    const int path = vec ? (long_rows && small ? 0 : 1) : 2;
    if (dtype == PLDP_BF16) {
        if (path == 0) return launch_pass_t<__nv_bfloat16, 0>(logits, a, scratch, s, what);
        if (path == 1) return launch_pass_t<__nv_bfloat16, 1>(logits, a, scratch, s, what);
        return launch_pass_t<__nv_bfloat16, 2>(logits, a, scratch, s, what);
    }
    if (path == 0) return launch_pass_t<float, 0>(logits, a, scratch, s, what);
    if (path == 1) return launch_pass_t<float, 1>(logits, a, scratch, s, what);
    return launch_pass_t<float, 2>(logits, a, scratch, s, what);
}

VerifyArgs verify_args(int B, int K, int V, const int32_t* draft, const int32_t* draft_len,
                       int32_t* argmax, int32_t* accept_len, int32_t* next_token, int32_t* ids,
                       int64_t ids_stride, int32_t* seq_len, int64_t T_cap, int32_t* kv_keep_len,
                       uint32_t* status) {
    VerifyArgs a = {};
    a.draft = draft;
    a.draft_len = draft_len;
    a.argmax = argmax;
    a.accept_len = accept_len;
    a.next_token = next_token;
    a.ids = ids;
    a.ids_stride = ids_stride;
    a.seq_len = seq_len;
    a.T_cap = T_cap;
    a.kv_keep_len = kv_keep_len;
    a.status = status;
    a.B = B;
    a.K = K;
    a.V = V;
    return a;
}


namespace {

// The pass, then the finish (one warp per sequence) behind its last wave.
pldp_status launch_verify(const void* logits, pldp_dtype dtype, const VerifyArgs& a0, void* scratch,
                          cudaStream_t s, const char* what) {
    VerifyArgs a = a0;
    const pldp_status st = launch_verify_pass(logits, dtype, a, scratch, s, what);
    if (st != PLDP_OK) return st;
    const unsigned fblocks = static_cast<unsigned>((a.B + kWarps - 1) / kWarps);
    const cudaError_t e = launch_pdl(verify_finish_kernel, dim3(fblocks), dim3(kThreads), 0, s, 0, a);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "%s: launch failed: %s", what, cudaGetErrorString(e));
    return PLDP_OK;
}

}  // namespace
}  // namespace pldp

using namespace pldp;

extern "C" PLDP_API size_t pldp_verify_workspace_size(int B, int K, int V) {
    if (B < 0 || K < 1 || V < 1) return 0;
    return keys_bytes(B, K);
}

extern "C" PLDP_API pldp_status pldp_extract_draft(const int32_t* ids, int64_t ids_stride,
                                                   const int32_t* seq_len, int64_t T_cap,
                                                   const int32_t* best_pos, int B, int K,
                                                   int32_t* draft, int32_t* draft_len,
                                                   void* stream) {
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "extract_draft: B < 0");
    if (K < 1) return fail(PLDP_ERR_INVALID_ARG, "extract_draft: K < 1");
    if (T_cap < 0 || T_cap > INT32_MAX) return fail(PLDP_ERR_INVALID_ARG, "extract_draft: bad T_cap");
    if (ids_stride < T_cap) return fail(PLDP_ERR_INVALID_ARG, "extract_draft: ids_stride < T_cap");
    if (B == 0) return PLDP_OK;
    if (!ids || !seq_len || !best_pos || !draft || !draft_len)
        return fail(PLDP_ERR_INVALID_ARG, "extract_draft: null pointer");
    const int64_t n = static_cast<int64_t>(B) * K;
    const int64_t blocks = (n + 255) / 256;
    if (blocks > INT32_MAX) return fail(PLDP_ERR_INVALID_ARG, "extract_draft: B*K too large");
    const cudaError_t e = launch_pdl(extract_draft_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0,
                                     static_cast<cudaStream_t>(stream), 0, ids, ids_stride, seq_len, T_cap,
                                     best_pos, B, K, draft, draft_len);
    if (e != cudaSuccess)
        return fail(PLDP_ERR_CUDA, "extract_draft: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}

extern "C" PLDP_API pldp_status pldp_verify_greedy(
    const void* logits, pldp_dtype dtype, int B, int K, int V, const int32_t* draft,
    const int32_t* draft_len, int32_t* argmax, int32_t* accept_len, int32_t* next_token,
    int32_t* ids, int64_t ids_stride, int32_t* seq_len, int64_t T_cap, int32_t* kv_keep_len,
    uint32_t* status, void* workspace, size_t workspace_bytes, void* stream) {
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy: B < 0");
    if (K < 1) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy: K < 1");
    if (V < 1) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy: V < 1");
    if (dtype != PLDP_F32 && dtype != PLDP_BF16)
        return fail(PLDP_ERR_UNSUPPORTED, "verify_greedy: unsupported dtype %d", (int)dtype);
    if ((ids || kv_keep_len) && !seq_len)
        return fail(PLDP_ERR_INVALID_ARG, "verify_greedy: ids/kv_keep_len need seq_len");
    if (seq_len && (T_cap < 0 || T_cap > INT32_MAX))
        return fail(PLDP_ERR_INVALID_ARG, "verify_greedy: bad T_cap");
    if (ids && ids_stride < T_cap) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy: ids_stride < T_cap");
    if (B == 0) return PLDP_OK;
    if (!logits || !draft || !draft_len || !accept_len || !next_token)
        return fail(PLDP_ERR_INVALID_ARG, "verify_greedy: null pointer");
    const size_t need = pldp_verify_workspace_size(B, K, V);
    if (!workspace || workspace_bytes < need)
        return fail(PLDP_ERR_INVALID_ARG, "verify_greedy: workspace needs %zu bytes", need);
    if (!aligned16(workspace)) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy: workspace not 16-byte aligned");

    const VerifyArgs a = verify_args(B, K, V, draft, draft_len, argmax, accept_len, next_token, ids,
                                     ids_stride, seq_len, T_cap, kv_keep_len, status);
    return launch_verify(logits, dtype, a, workspace, static_cast<cudaStream_t>(stream),
                         "verify_greedy");
}

// ---------------------------------------------------------------------------
// Sampling verification (Sec. 4.4 at temperature T > 0).
//
// Position i of sequence b draws the smallest v whose cumulative probability
// under p = softmax(logits[b, i] / T) exceeds the caller's uniform u[b, i]
// (inverse-CDF sampling); the draft is then accepted up to the first position
// whose draw differs from it, and the draw there is the bonus -- for a
// single-token-per-position draft this is exactly what sampling from the target
// would emit.
//
// 1. A stats pass streams the logits once, in the same moving-window order as
//    the greedy pass, over units of (row, 2 KB piece): per piece the max M_k and
//    S_k = sum 2^((l - M_k) log2(e) / T).  No atomics: each piece has its slot.
// 2. One CTA per sequence, one warp per row: the piece weights
//    W_k = S_k 2^((M_k - M) log2(e) / T) against the row max M give the total Z
//    (a warp scan over the pieces, run twice in the same order, so the second
//    run's crossing of u Z always exists), which picks the piece; the warp then
//    rereads that one piece and finds the element where the running sum of its
//    weights passes the same fraction of the piece.  fp32 throughout: a draw can
//    differ from the exact one only when u lies within rounding (~1e-6) of a
//    boundary of the cumulative distribution.
// ---------------------------------------------------------------------------
namespace pldp {
namespace {

constexpr int64_t kPieceBytes = 2048;

struct SampleArgs {
    VerifyArgs v;                   // draft, bookkeeping; v.argmax receives the draws
    const float* uniforms;          // [B*(K+1)]
    const float2* stats;            // [rows * npieces]: (M_k, S_k)
    float c;                        // log2(e) / T
    int npieces;                    // pieces per row
    int P;                          // elements per piece
};

__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// The elements of one 16-byte vector as floats.
__device__ __forceinline__ void unpack(const uint4& x, float (&e)[8], __nv_bfloat16) {
    const uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        e[2 * k] = __uint_as_float(w[k] << 16);
        e[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
    }
}
__device__ __forceinline__ void unpack(const uint4& x, float (&e)[8], float) {
    e[0] = __uint_as_float(x.x);
    e[1] = __uint_as_float(x.y);
    e[2] = __uint_as_float(x.z);
    e[3] = __uint_as_float(x.w);
}

__device__ __forceinline__ float warp_max_f(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
    return v;
}

// The float of an ordered key (inverse of ordered_key).
__device__ __forceinline__ float ordered_value(uint32_t o) {
    return __uint_as_float((o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o);
}

// 1. per-piece (max, sum of weights).  Units u = row * npieces + piece, warp w of W
// takes units w, w + W, ...; piece k of row r covers elements [k P, min((k+1) P, V)).
// Each lane sums its elements' weights against its own maximum m, so the
// exponentials do not wait for the piece's maximum M (one redux over ordered
// keys); the lane's sum is then scaled by 2^((m - M) / T log2 e) and the warp adds.
template <typename T, bool VEC>
__global__ void __launch_bounds__(kThreads, VEC ? kPassBlocksPerSm : 4)
sample_stats_kernel(const T* __restrict__ logits, int64_t V, int64_t rows, int npieces, int P, float c,
                    int64_t W, float2* __restrict__ stats) {
    pdl_wait_only();                        // the finish (a full SM per CTA) starts as this grid ends
    const int lane = threadIdx.x & 31;
    const int64_t w = static_cast<int64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
    const int64_t units = rows * npieces;
    int64_t r = w / npieces, k = w - r * npieces;
    const int64_t dr = W / npieces, dk = W - dr * npieces;
    for (int64_t u = w; u < units; u += W) {
        const int64_t e0 = static_cast<int64_t>(k) * P;
        const int64_t n = (V - e0 < P) ? V - e0 : P;            // elements in this piece
        const T* piece = logits + r * V + e0;
        float m = -INFINITY, sum = 0.f, M;
        if constexpr (VEC) {
            // whole 16-byte vectors: V, hence every piece length, is a multiple of one
            constexpr int VW = 16 / static_cast<int>(sizeof(T));
            const uint4* pv = reinterpret_cast<const uint4*>(piece);
            uint4 raw[kSegLoads];
#pragma unroll
            for (int q = 0; q < kSegLoads; ++q) {
                const int vi = lane + 32 * q;
                if (static_cast<int64_t>(vi) * VW < n) raw[q] = ld_stream16(pv + vi);
            }
#pragma unroll
            for (int q = 0; q < kSegLoads; ++q)
                if (static_cast<int64_t>(lane + 32 * q) * VW < n) m = fmaxf(m, vmax(raw[q], T()));
            if (m > -INFINITY) {
                const float mc = m * c;
#pragma unroll
                for (int q = 0; q < kSegLoads; ++q) {
                    if (static_cast<int64_t>(lane + 32 * q) * VW >= n) continue;
                    float e[8];
                    unpack(raw[q], e, T());
#pragma unroll
                    for (int j = 0; j < VW; j += 2)                // pairs: half the dependent adds
                        sum += ex2_approx(fmaf(e[j], c, -mc)) + ex2_approx(fmaf(e[j + 1], c, -mc));
                }
            }
            M = ordered_value(__reduce_max_sync(0xFFFFFFFFu, ordered_key(m)));
            if (sum > 0.f) sum *= ex2_approx((m - M) * c);
        } else {
            constexpr int PER = static_cast<int>(kPieceBytes / sizeof(T)) / 32;
            float x[PER];
#pragma unroll
            for (int q = 0; q < PER; ++q) {
                const int ei = lane + 32 * q;
                x[q] = ei < n ? to_f32(piece[ei]) : -INFINITY;
                m = fmaxf(m, x[q]);
            }
            if (m > -INFINITY) {
                const float mc = m * c;
#pragma unroll
                for (int q = 0; q < PER; ++q)
                    if (x[q] > -INFINITY) sum += ex2_approx(fmaf(x[q], c, -mc));
            }
            M = ordered_value(__reduce_max_sync(0xFFFFFFFFu, ordered_key(m)));
            if (sum > 0.f) sum *= ex2_approx((m - M) * c);
        }
        sum = warp_sum(sum);
        if (lane == 0) stats[u] = make_float2(M, sum);
        r += dr;
        k += dk;
        if (k >= npieces) {
            k -= npieces;
            ++r;
        }
    }
}

// Weight of piece k of a row against the row max M (0 for an empty piece).
__device__ __forceinline__ float piece_weight(const float2* st, int k, int npieces, float Mc, float c) {
    if (k >= npieces) return 0.f;
    const float2 s = __ldcg(st + k);
    return s.x > -INFINITY ? s.y * ex2_approx(fmaf(s.x, c, -Mc)) : 0.f;
}

__device__ __forceinline__ float warp_incl_scan(float v, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float t = __shfl_up_sync(0xFFFFFFFFu, v, o);
        if (lane >= o) v += t;
    }
    return v;
}

// Piece k* of row r, where the running total of the piece weights first passes
// u Z: the total is summed, then the crossing found, by the same warp scans in the
// same order, so the crossing exists.  The row's stats are held in registers
// (up to 32 * kStatRegs pieces) or, beyond that, reread per scan.
constexpr int kStatRegs = 4;

struct PiecePick {
    int k;          // the piece
    float before;   // running total before it
    float w;        // its weight
    float target;   // u Z
    float Mk;       // its max
};

__device__ __forceinline__ PiecePick pick_piece(const float2* __restrict__ st, int np, float c, float u, int lane) {
    PiecePick pk = {-1, 0.f, 0.f, 0.f, 0.f};
    if (np <= 32 * kStatRegs) {
        float2 sv[kStatRegs];
        float m = -INFINITY;
#pragma unroll
        for (int q = 0; q < kStatRegs; ++q) {
            const int k = lane + 32 * q;
            sv[q] = k < np ? __ldcg(st + k) : make_float2(-INFINITY, 0.f);
            m = fmaxf(m, sv[q].x);
        }
        const float Mc = warp_max_f(m) * c;
        float wv[kStatRegs], incl[kStatRegs], total = 0.f;
#pragma unroll
        for (int q = 0; q < kStatRegs; ++q) {
            wv[q] = sv[q].x > -INFINITY ? sv[q].y * ex2_approx(fmaf(sv[q].x, c, -Mc)) : 0.f;
            incl[q] = warp_incl_scan(wv[q], lane);
            total += __shfl_sync(0xFFFFFFFFu, incl[q], 31);
        }
        pk.target = u * total;
        float run = 0.f;
#pragma unroll
        for (int q = 0; q < kStatRegs; ++q) {
            const unsigned hit = __ballot_sync(0xFFFFFFFFu, run + incl[q] > pk.target && lane + 32 * q < np);
            if (pk.k < 0 && hit) {
                const int f = __ffs(hit) - 1;
                pk.k = 32 * q + f;
                pk.before = run + __shfl_sync(0xFFFFFFFFu, incl[q] - wv[q], f);
                pk.w = __shfl_sync(0xFFFFFFFFu, wv[q], f);
                pk.Mk = __shfl_sync(0xFFFFFFFFu, sv[q].x, f);
            }
            run += __shfl_sync(0xFFFFFFFFu, incl[q], 31);
        }
    } else {
        float m = -INFINITY;
        for (int k = lane; k < np; k += 32) m = fmaxf(m, __ldcg(st + k).x);
        const float Mc = warp_max_f(m) * c;
        float total = 0.f;
        for (int k0 = 0; k0 < np; k0 += 32) {
            const float incl = warp_incl_scan(piece_weight(st, k0 + lane, np, Mc, c), lane);
            total += __shfl_sync(0xFFFFFFFFu, incl, 31);
        }
        pk.target = u * total;
        float run = 0.f;
        for (int k0 = 0; k0 < np && pk.k < 0; k0 += 32) {
            const float wv = piece_weight(st, k0 + lane, np, Mc, c);
            const float incl = warp_incl_scan(wv, lane);
            const unsigned hit = __ballot_sync(0xFFFFFFFFu, run + incl > pk.target && k0 + lane < np);
            if (hit) {
                const int f = __ffs(hit) - 1;
                pk.k = k0 + f;
                pk.before = run + __shfl_sync(0xFFFFFFFFu, incl - wv, f);
                pk.w = __shfl_sync(0xFFFFFFFFu, wv, f);
                pk.Mk = __ldcg(st + pk.k).x;
            }
            run += __shfl_sync(0xFFFFFFFFu, incl, 31);
        }
    }
    return pk;
}

// The draw of row r (one warp).
template <typename T, bool VEC>
__device__ int sample_row(const T* __restrict__ logits, const SampleArgs& a, int64_t r, int lane) {
    const int64_t V = a.v.V;
    const int np = a.npieces;
    const float2* st = a.stats + r * np;
    float u = a.uniforms[r];
    if (!(u >= 0.f)) u = 0.f;
    if (u >= 1.f) u = __uint_as_float(0x3F7FFFFFu);               // largest float below 1
    PiecePick pk = pick_piece(st, np, a.c, u, lane);
    float f;                                                      // fraction of the piece to pass
    if (pk.k < 0) {
        // u Z rounded up to Z (u within 2^-24 of 1): the end of the last piece with weight
        int k = np - 1;
        for (; k > 0; --k)
            if (__ldcg(st + k).y > 0.f) break;
        pk.k = k;
        pk.Mk = __ldcg(st + k).x;
        f = 1.f;
    } else {
        f = pk.w > 0.f ? (pk.target - pk.before) / pk.w : 0.f;
    }
    f = fminf(fmaxf(f, 0.f), __uint_as_float(0x3F7FFFFFu));
    const int ks = pk.k;
    // the piece, lane L holding its elements [L E, (L+1) E) in index order
    constexpr int E = static_cast<int>(kPieceBytes / sizeof(T)) / 32;
    const int64_t e0 = static_cast<int64_t>(ks) * a.P;
    const int64_t n = (V - e0 < a.P) ? V - e0 : a.P;
    const T* piece = logits + r * V + e0;
    const float Mkc = pk.Mk * a.c;
    float x[E];
    if constexpr (VEC) {
        constexpr int VW = 16 / static_cast<int>(sizeof(T));
        const uint4* pv = reinterpret_cast<const uint4*>(piece) + lane * (E / VW);
#pragma unroll
        for (int q = 0; q < E / VW; ++q) {
            const int64_t ei = static_cast<int64_t>(lane) * E + q * VW;
            uint4 raw = make_uint4(0u, 0u, 0u, 0u);
            if (ei < n) raw = __ldcg(pv + q);
            float e[8];
            unpack(raw, e, T());
#pragma unroll
            for (int j = 0; j < VW; ++j) x[q * VW + j] = ei + j < n ? e[j] : -INFINITY;
        }
    } else {
#pragma unroll
        for (int q = 0; q < E; ++q) {
            const int64_t ei = static_cast<int64_t>(lane) * E + q;
            x[q] = ei < n ? to_f32(piece[ei]) : -INFINITY;
        }
    }
    float ls = 0.f;
#pragma unroll
    for (int j = 0; j < E; ++j) ls += x[j] > -INFINITY ? ex2_approx(fmaf(x[j], a.c, -Mkc)) : 0.f;
    const float incl = warp_incl_scan(ls, lane);
    const float tot = __shfl_sync(0xFFFFFFFFu, incl, 31);
    const float tgt = f * tot;
    const unsigned hit = __ballot_sync(0xFFFFFFFFu, incl > tgt && ls > 0.f);
    const unsigned has = __ballot_sync(0xFFFFFFFFu, ls > 0.f);
    // the lane where the running sum passes the target; if rounding hides it, the
    // last lane holding weight (its last element with weight is then drawn)
    const int L0 = hit ? __ffs(hit) - 1 : (has ? 31 - __clz(has) : 0);
    int y = -1;
    if (lane == L0) {
        float acc = incl - ls;
        int last = -1;
#pragma unroll
        for (int j = 0; j < E; ++j) {
            const float wv = x[j] > -INFINITY ? ex2_approx(fmaf(x[j], a.c, -Mkc)) : 0.f;
            if (wv > 0.f) last = j;
            acc += wv;
            if (y < 0 && acc > tgt) y = j;
        }
        if (y < 0) y = last;                                      // rounding inside the lane
        if (y < 0) y = 0;
        y = static_cast<int>(static_cast<int64_t>(L0) * E + y + e0);
    }
    return __shfl_sync(0xFFFFFFFFu, y, L0);
}

// 2. draws and acceptance: one CTA per sequence, warp w draws rows w, w + 16, ...
constexpr int kFinishWarps = 16;

template <typename T, bool VEC>
__global__ void __launch_bounds__(32 * kFinishWarps, 1) sample_finish_kernel(const T* __restrict__ logits,
                                                                            SampleArgs a) {
    extern __shared__ int32_t draws[];                           // [K+1]
    pdl_enter();
    const int64_t b = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int K1 = a.v.K + 1;
    if (warp == kFinishWarps - 1) {                              // what the finish reads, on its way to L1
        for (int i = lane; i < a.v.K; i += 32)
            asm volatile("prefetch.global.L1 [%0];" ::"l"(a.v.draft + b * a.v.K + i));
        if (lane == 0) asm volatile("prefetch.global.L1 [%0];" ::"l"(a.v.draft_len + b));
        if (lane == 1 && a.v.seq_len) asm volatile("prefetch.global.L1 [%0];" ::"l"(a.v.seq_len + b));
    }
    for (int i = warp; i < K1; i += kFinishWarps) {
        const int y = sample_row<T, VEC>(logits, a, b * K1 + i, lane);
        if (lane == 0) draws[i] = y;
    }
    __syncthreads();
    if (warp == 0) finish_sequence(a.v, b, lane, SharedTokens{draws});
}

int sample_pieces(int V, size_t es) {
    const int64_t P = kPieceBytes / static_cast<int64_t>(es);
    return static_cast<int>((V + P - 1) / P);
}

template <typename T, bool VEC>
pldp_status launch_sample_t(const void* logits, SampleArgs a, cudaStream_t s) {
    const int64_t rows = static_cast<int64_t>(a.v.B) * (a.v.K + 1);
    const int64_t units = rows * a.npieces;
    const void* fn = reinterpret_cast<const void*>(&sample_stats_kernel<T, VEC>);
    int64_t blocks = static_cast<int64_t>(resident_blocks(fn, kThreads, 0)) * kPassWaves;
    const int64_t need = (units + kWarps - 1) / kWarps;
    if (blocks > need) blocks = need;
    if (blocks < 1) blocks = 1;
    cudaError_t e = launch_pdl(sample_stats_kernel<T, VEC>, dim3(static_cast<unsigned>(blocks)), dim3(kThreads), 0,
                               s, 0, static_cast<const T*>(logits), static_cast<int64_t>(a.v.V), rows, a.npieces,
                               a.P, a.c, blocks * kWarps, const_cast<float2*>(a.stats));
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "verify_sample: launch failed: %s", cudaGetErrorString(e));
    const size_t smem = static_cast<size_t>(a.v.K + 1) * sizeof(int32_t);
    if (smem > 48 * 1024) {
        e = cudaFuncSetAttribute(sample_finish_kernel<T, VEC>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(smem));
        if (e != cudaSuccess)
            return fail(PLDP_ERR_CUDA, "verify_sample: shared memory attribute: %s", cudaGetErrorString(e));
    }
    e = launch_pdl(sample_finish_kernel<T, VEC>, dim3(static_cast<unsigned>(a.v.B)), dim3(32 * kFinishWarps), smem, s, 0,
                   static_cast<const T*>(logits), a);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "verify_sample: launch failed: %s", cudaGetErrorString(e));
    return PLDP_OK;
}

}  // namespace
}  // namespace pldp

extern "C" PLDP_API size_t pldp_verify_sample_workspace_size(int B, int K, int V, pldp_dtype dtype) {
    if (B < 0 || K < 1 || V < 1 || (dtype != PLDP_F32 && dtype != PLDP_BF16)) return 0;
    const size_t es = dtype == PLDP_F32 ? 4 : 2;
    const size_t bytes = static_cast<size_t>(B) * (K + 1) * sample_pieces(V, es) * sizeof(float2);
    return (bytes + 255) / 256 * 256;
}

extern "C" PLDP_API pldp_status pldp_verify_sample(
    const void* logits, pldp_dtype dtype, int B, int K, int V, float temperature, const float* uniforms,
    const int32_t* draft, const int32_t* draft_len, int32_t* sampled, int32_t* accept_len, int32_t* next_token,
    int32_t* ids, int64_t ids_stride, int32_t* seq_len, int64_t T_cap, int32_t* kv_keep_len, uint32_t* status,
    void* workspace, size_t workspace_bytes, void* stream) {
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "verify_sample: B < 0");
    if (K < 1) return fail(PLDP_ERR_INVALID_ARG, "verify_sample: K < 1");
    if (V < 1) return fail(PLDP_ERR_INVALID_ARG, "verify_sample: V < 1");
    if (dtype != PLDP_F32 && dtype != PLDP_BF16)
        return fail(PLDP_ERR_UNSUPPORTED, "verify_sample: unsupported dtype %d", (int)dtype);
    if (!(temperature > 0.f) || isinf(temperature))
        return fail(PLDP_ERR_INVALID_ARG, "verify_sample: temperature must be positive and finite");
    if ((ids || kv_keep_len) && !seq_len)
        return fail(PLDP_ERR_INVALID_ARG, "verify_sample: ids/kv_keep_len need seq_len");
    if (seq_len && (T_cap < 0 || T_cap > INT32_MAX)) return fail(PLDP_ERR_INVALID_ARG, "verify_sample: bad T_cap");
    if (ids && ids_stride < T_cap) return fail(PLDP_ERR_INVALID_ARG, "verify_sample: ids_stride < T_cap");
    if (static_cast<int64_t>(K) + 1 > 12288) return fail(PLDP_ERR_UNSUPPORTED, "verify_sample: K > 12287");
    if (B == 0) return PLDP_OK;
    if (!logits || !uniforms || !draft || !draft_len || !accept_len || !next_token)
        return fail(PLDP_ERR_INVALID_ARG, "verify_sample: null pointer");
    const size_t need = pldp_verify_sample_workspace_size(B, K, V, dtype);
    if (!workspace || workspace_bytes < need)
        return fail(PLDP_ERR_INVALID_ARG, "verify_sample: workspace needs %zu bytes", need);
    if (!aligned16(workspace)) return fail(PLDP_ERR_INVALID_ARG, "verify_sample: workspace not 16-byte aligned");

    const size_t es = dtype == PLDP_F32 ? 4 : 2;
    SampleArgs a = {};
    a.v = verify_args(B, K, V, draft, draft_len, sampled, accept_len, next_token, ids, ids_stride, seq_len, T_cap,
                      kv_keep_len, status);
    a.uniforms = uniforms;
    a.stats = static_cast<const float2*>(workspace);
    a.c = 1.4426950408889634f / temperature;                      // log2(e) / T
    a.npieces = sample_pieces(V, es);
    a.P = static_cast<int>(kPieceBytes / static_cast<int64_t>(es));
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const bool vec = aligned16(logits) && (static_cast<size_t>(V) * es) % 16 == 0;
    if (dtype == PLDP_BF16)
        return vec ? launch_sample_t<__nv_bfloat16, true>(logits, a, s) : launch_sample_t<__nv_bfloat16, false>(logits, a, s);
    return vec ? launch_sample_t<float, true>(logits, a, s) : launch_sample_t<float, false>(logits, a, s);
}

// ---------------------------------------------------------------------------
// Allocation-free greedy verification.
//
// Some callers cannot hand the library a workspace: code that owns no device
// allocator (a plugin living inside a host program that manages all GPU memory
// itself), and serving loops that forbid cudaMalloc/cudaFree once they are up,
// because those calls can synchronise the device and stall every stream.  For
// them this entry point keeps its scratch in a fixed area compiled into the
// library.  Every GPU that loads the library holds that area until the process
// exits.
// ---------------------------------------------------------------------------
#include <mutex>

namespace pldp {
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(1) << 20;   // 1 MiB: B*(K+1) up to ~130k rows
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mutex;
void* g_noalloc_ptr[kMaxDevices] = {};

// Device address of g_noalloc_scratch on the current device, looked up once per
// device.  In host code the array's name only stands in for the symbol; the
// kernel must be given this address instead.
pldp_status noalloc_scratch(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return fail(PLDP_ERR_CUDA, "verify_greedy_noalloc: cudaGetDevice: %s", cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDevices)
        return fail(PLDP_ERR_UNSUPPORTED, "verify_greedy_noalloc: device %d beyond %d", dev, kMaxDevices);
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (!g_noalloc_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p)
            return fail(PLDP_ERR_CUDA, "verify_greedy_noalloc: cudaGetSymbolAddress: %s",
                        cudaGetErrorString(e));
        g_noalloc_ptr[dev] = p;
    }
    *out = g_noalloc_ptr[dev];
    return PLDP_OK;
}

}  // namespace
}  // namespace pldp

extern "C" PLDP_API pldp_status pldp_verify_greedy_noalloc(
    const void* logits, pldp_dtype dtype, int B, int K, int V, const int32_t* draft,
    const int32_t* draft_len, int32_t* argmax, int32_t* accept_len, int32_t* next_token,
    int32_t* ids, int64_t ids_stride, int32_t* seq_len, int64_t T_cap, int32_t* kv_keep_len,
    uint32_t* status, void* stream) {
    if (B < 0) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_noalloc: B < 0");
    if (K < 1) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_noalloc: K < 1");
    if (V < 1) return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_noalloc: V < 1");
    if (dtype != PLDP_F32 && dtype != PLDP_BF16)
        return fail(PLDP_ERR_UNSUPPORTED, "verify_greedy_noalloc: unsupported dtype %d", (int)dtype);
    if ((ids || kv_keep_len) && !seq_len)
        return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_noalloc: ids/kv_keep_len need seq_len");
    if (seq_len && (T_cap < 0 || T_cap > INT32_MAX))
        return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_noalloc: bad T_cap");
    if (ids && ids_stride < T_cap)
        return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_noalloc: ids_stride < T_cap");
    const size_t need = pldp_verify_workspace_size(B, K, V);
    if (need > kNoAllocScratchBytes)
        return fail(PLDP_ERR_INVALID_ARG,
                    "verify_greedy_noalloc: B=%d, K=%d needs %zu bytes of scratch; the built-in area "
                    "holds %zu (use pldp_verify_greedy with a caller workspace)",
                    B, K, need, kNoAllocScratchBytes);
    if (B == 0) return PLDP_OK;
    if (!logits || !draft || !draft_len || !accept_len || !next_token)
        return fail(PLDP_ERR_INVALID_ARG, "verify_greedy_noalloc: null pointer");

    void* scratch = nullptr;
    pldp_status ps = noalloc_scratch(&scratch);
    if (ps != PLDP_OK) return ps;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // The kernels need the row keys at zero.  Each call returns them to zero when
    // it completes, but the area is shared and outlives every call, so it is
    // cleared here as well (cudaMemsetAsync allocates nothing).
    cudaError_t e = cudaMemsetAsync(scratch, 0, need, s);
    if (e != cudaSuccess)
        return fail(PLDP_ERR_CUDA, "verify_greedy_noalloc: clearing scratch: %s", cudaGetErrorString(e));

    const VerifyArgs a = verify_args(B, K, V, draft, draft_len, argmax, accept_len, next_token, ids,
                                     ids_stride, seq_len, T_cap, kv_keep_len, status);
    return launch_verify(logits, dtype, a, scratch, s, "verify_greedy_noalloc");
}
