// Draft prediction (Sec. 4.3) and greedy verification (Sec. 4.4) of PLD+.
//
// Verification is two kernels chained by programmatic dependent launch.
//
// 1. One streaming pass over the flattened logits [B, K+1, V], cut into 2 KB
//    segments.  Warp w of the W in the grid takes segments w, w + W, w + 2W, ...
//    so the segments in flight form a moving window over memory, and the grid
//    is many waves of small CTAs, so the block scheduler keeps every SM busy to
//    the end (faster SMs take more CTAs).  Each lane issues its four 16-byte
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
constexpr int kPassWaves = 11;              // grid = up to 11 waves of resident CTAs

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
// than segments) and launches it.  `a` has everything but the keys.  At the
// sustained-loop shape 11 waves (about two segments per warp) measured best,
// alternated on one box: verification 66.0-66.1 us against 67.4-67.8 us for 6
// waves and 66.9-67.2 us for exactly two segments per warp; 4, 8, 10, 12-16 and
// 24 waves, and one segment per warp, measured slower.
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
namespace pldp {
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(1) << 20;   // 1 MiB: B*(K+1) up to ~130k rows

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of g_noalloc_scratch in the CUDA context current on this thread.
// In host code the array's name only stands in for the symbol; the kernels must
// be given this address instead.  It is looked up on every call, not cached: the
// address belongs to a context, and a caller may switch contexts or reset the
// device between calls.  cudaGetSymbolAddress allocates nothing.
pldp_status noalloc_scratch(void** out) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess || !p)
        return fail(PLDP_ERR_CUDA, "verify_greedy_noalloc: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
    *out = p;
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
