// Sampling verification of PLD+ (Sec. 4.4 at temperature T > 0): pldp_verify_sample.
#include <math.h>

#include "pldp_internal.cuh"
#include "pldp_verify.cuh"

namespace pldp {
namespace {

// The streaming shape of the greedy pass (verify.cu): 256-thread CTAs, 2 KB per warp
// and unit (four 16-byte loads per lane), up to 11 waves of 8 CTAs per SM.  At the
// sustained-loop shape, alternated on one box with the spill-free kernel below:
// 11 waves 67.9 us per call, 6 waves 69.3 us, 4 waves 71.2 us.
constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kSegLoads = 4;
constexpr int kPassBlocksPerSm = 8;
constexpr int kPassWaves = 11;

}  // namespace
}  // namespace pldp

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

// Two floats in one 64-bit register pair, and the packed fp32 operations on them
// (one instruction for two lanes of fp32 FMA or add): the stats pass weighs its
// elements two at a time.
__device__ __forceinline__ uint64_t pack_f32x2(float lo, float hi) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ float lo_f32(uint64_t x) {
    float lo, hi;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(x));
    return lo;
}
__device__ __forceinline__ float hi_f32(uint64_t x) {
    float lo, hi;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(x));
    return hi;
}
__device__ __forceinline__ uint64_t fma_f32x2(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
__device__ __forceinline__ uint64_t add_f32x2(uint64_t a, uint64_t b) {
    uint64_t d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
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
//
// The streaming form: 16-byte loads (every piece a whole number of vectors) and
// 32-bit unit arithmetic (fewer than 2^31 units, checked on the host; the rows and
// pieces a grid stride advances come from the host), which keeps the kernel within
// the 32 registers of 8 CTAs per SM without spilling: 72.2 -> 69.5 us per call at
// the sustained-loop shape against the earlier 64-bit form, which spilled.  Each
// lane's weights are summed in even/odd pairs with packed fp32 FMA and add.
template <typename T>
__global__ void __launch_bounds__(kThreads, kPassBlocksPerSm)
sample_stats_vec_kernel(const T* __restrict__ logits, uint32_t V, uint32_t units, uint32_t npieces, uint32_t P,
                        float c, uint32_t W, uint32_t dr, uint32_t dk, float2* __restrict__ stats) {
    // W = warps in the grid = dr rows and dk pieces
    pdl_wait_only();                        // the finish (a full SM per CTA) starts as this grid ends
    constexpr uint32_t VW = 16 / sizeof(T);
    const int lane = threadIdx.x & 31;
    const uint32_t w = blockIdx.x * kWarps + (threadIdx.x >> 5);
    uint32_t r = w / npieces, k = w - r * npieces;
    for (uint32_t u = w; u < units; u += W) {
        const uint32_t e0 = k * P;
        const uint32_t nv = (V - e0 < P ? V - e0 : P) / VW;            // vectors in this piece
        const uint4* pv = reinterpret_cast<const uint4*>(logits + (static_cast<uint64_t>(r) * V + e0));
        uint4 raw[kSegLoads];
#pragma unroll
        for (int q = 0; q < kSegLoads; ++q)
            if (lane + 32u * q < nv) raw[q] = ld_stream16(pv + lane + 32 * q);
        float m = -INFINITY, sum = 0.f;
#pragma unroll
        for (int q = 0; q < kSegLoads; ++q)
            if (lane + 32u * q < nv) m = fmaxf(m, vmax(raw[q], T()));
        if (m > -INFINITY) {
            const float mc = m * c;
            const uint64_t c2 = pack_f32x2(c, c), mc2 = pack_f32x2(-mc, -mc);
            uint64_t acc = 0;                                          // (0.f, 0.f)
#pragma unroll
            for (int q = 0; q < kSegLoads; ++q) {
                if (lane + 32u * q >= nv) continue;
                float e[8];
                unpack(raw[q], e, T());
#pragma unroll
                for (int j = 0; j < static_cast<int>(VW); j += 2) {    // element pairs, packed fp32 math
                    const uint64_t x = fma_f32x2(pack_f32x2(e[j], e[j + 1]), c2, mc2);
                    acc = add_f32x2(acc, pack_f32x2(ex2_approx(lo_f32(x)), ex2_approx(hi_f32(x))));
                }
            }
            sum = lo_f32(acc) + hi_f32(acc);
        }
        const float M = ordered_value(__reduce_max_sync(0xFFFFFFFFu, ordered_key(m)));
        if (sum > 0.f) sum *= ex2_approx((m - M) * c);
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

// The element-load form, for unaligned logits or rows that are not a whole number
// of 16-byte vectors.
template <typename T>
__global__ void __launch_bounds__(kThreads, 4)
sample_stats_kernel(const T* __restrict__ logits, int64_t V, int64_t rows, int npieces, int P, float c,
                    int64_t W, float2* __restrict__ stats) {
    pdl_wait_only();
    const int lane = threadIdx.x & 31;
    const int64_t w = static_cast<int64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
    const int64_t units = rows * npieces;
    int64_t r = w / npieces, k = w - r * npieces;
    const int64_t dr = W / npieces, dk = W - dr * npieces;
    for (int64_t u = w; u < units; u += W) {
        const int64_t e0 = static_cast<int64_t>(k) * P;
        const int64_t n = (V - e0 < P) ? V - e0 : P;            // elements in this piece
        const T* piece = logits + r * V + e0;
        float m = -INFINITY, sum = 0.f;
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
        const float M = ordered_value(__reduce_max_sync(0xFFFFFFFFu, ordered_key(m)));
        if (sum > 0.f) sum *= ex2_approx((m - M) * c);
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

// Draws only, for the fused sampling + next draft call: one warp per row, each
// draw to draws[row]; the accept/bonus/append and the drafting follow in the
// next kernel.
template <typename T, bool VEC>
__global__ void __launch_bounds__(kThreads) sample_draw_kernel(const T* __restrict__ logits, SampleArgs a,
                                                                int32_t* __restrict__ draws) {
    pdl_enter();
    const int64_t r = static_cast<int64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5);   // warp-uniform
    const int64_t rows = static_cast<int64_t>(a.v.B) * (a.v.K + 1);
    if (r >= rows) return;
    const int y = sample_row<T, VEC>(logits, a, r, threadIdx.x & 31);
    if ((threadIdx.x & 31) == 0) draws[r] = y;
}

int sample_pieces(int V, size_t es) {
    const int64_t P = kPieceBytes / static_cast<int64_t>(es);
    return static_cast<int>((V + P - 1) / P);
}

template <typename T, bool VEC>
pldp_status launch_stats_t(const void* logits, const SampleArgs& a, cudaStream_t s, const char* what) {
    const int64_t rows = static_cast<int64_t>(a.v.B) * (a.v.K + 1);
    const int64_t units = rows * a.npieces;
    const bool vec = VEC && units < (int64_t(1) << 31);               // 32-bit unit arithmetic
    const void* fn = vec ? reinterpret_cast<const void*>(&sample_stats_vec_kernel<T>)
                         : reinterpret_cast<const void*>(&sample_stats_kernel<T>);
    int64_t blocks = static_cast<int64_t>(resident_blocks(fn, kThreads, 0)) * kPassWaves;
    const int64_t need = (units + kWarps - 1) / kWarps;
    if (blocks > need) blocks = need;
    if (blocks < 1) blocks = 1;
    const T* lp = static_cast<const T*>(logits);
    float2* st = const_cast<float2*>(a.stats);
    const cudaError_t e =
        vec ? launch_pdl(sample_stats_vec_kernel<T>, dim3(static_cast<unsigned>(blocks)), dim3(kThreads), 0, s, 0, lp,
                         static_cast<uint32_t>(a.v.V), static_cast<uint32_t>(units), static_cast<uint32_t>(a.npieces),
                         static_cast<uint32_t>(a.P), a.c, static_cast<uint32_t>(blocks * kWarps),
                         static_cast<uint32_t>(blocks * kWarps / a.npieces),
                         static_cast<uint32_t>(blocks * kWarps % a.npieces), st)
            : launch_pdl(sample_stats_kernel<T>, dim3(static_cast<unsigned>(blocks)), dim3(kThreads), 0, s, 0, lp,
                         static_cast<int64_t>(a.v.V), rows, a.npieces, a.P, a.c, blocks * kWarps, st);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "%s: launch failed: %s", what, cudaGetErrorString(e));
    return PLDP_OK;
}

template <typename T, bool VEC>
pldp_status launch_draws_t(const void* logits, const SampleArgs& a, int32_t* draws, cudaStream_t s,
                           const char* what) {
    const pldp_status st = launch_stats_t<T, VEC>(logits, a, s, what);
    if (st != PLDP_OK) return st;
    const int64_t rows = static_cast<int64_t>(a.v.B) * (a.v.K + 1);
    const cudaError_t e = launch_pdl(sample_draw_kernel<T, VEC>, dim3(static_cast<unsigned>((rows + kWarps - 1) / kWarps)),
                                     dim3(kThreads), 0, s, 0, static_cast<const T*>(logits), a, draws);
    if (e != cudaSuccess) return fail(PLDP_ERR_CUDA, "%s: launch failed: %s", what, cudaGetErrorString(e));
    return PLDP_OK;
}

template <typename T, bool VEC>
pldp_status launch_sample_t(const void* logits, SampleArgs a, cudaStream_t s) {
    const pldp_status st = launch_stats_t<T, VEC>(logits, a, s, "verify_sample");
    if (st != PLDP_OK) return st;
    cudaError_t e;
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

namespace pldp {

size_t sample_draft_workspace_size(int B, int K, int V, pldp_dtype dtype) {
    if (B < 0 || K < 1 || V < 1 || (dtype != PLDP_F32 && dtype != PLDP_BF16)) return 0;
    const size_t es = dtype == PLDP_F32 ? 4 : 2;
    const size_t rows = static_cast<size_t>(B) * (K + 1);
    const size_t stats = (rows * sample_pieces(V, es) * sizeof(float2) + 255) / 256 * 256;
    return stats + (rows * sizeof(int32_t) + 255) / 256 * 256;
}

pldp_status launch_sample_draws(const void* logits, pldp_dtype dtype, VerifyArgs& v, float temperature,
                                const float* uniforms, void* workspace, cudaStream_t s, const char* what) {
    const size_t es = dtype == PLDP_F32 ? 4 : 2;
    const size_t rows = static_cast<size_t>(v.B) * (v.K + 1);
    SampleArgs a = {};
    a.v = v;
    a.uniforms = uniforms;
    a.stats = static_cast<const float2*>(workspace);
    a.c = 1.4426950408889634f / temperature;                      // log2(e) / T
    a.npieces = sample_pieces(v.V, es);
    a.P = static_cast<int>(kPieceBytes / static_cast<int64_t>(es));
    int32_t* draws = reinterpret_cast<int32_t*>(static_cast<char*>(workspace) +
                                                (rows * a.npieces * sizeof(float2) + 255) / 256 * 256);
    v.row_draws = draws;
    const bool vec = aligned16(logits) && (static_cast<size_t>(v.V) * es) % 16 == 0;
    if (dtype == PLDP_BF16)
        return vec ? launch_draws_t<__nv_bfloat16, true>(logits, a, draws, s, what)
                   : launch_draws_t<__nv_bfloat16, false>(logits, a, draws, s, what);
    return vec ? launch_draws_t<float, true>(logits, a, draws, s, what)
               : launch_draws_t<float, false>(logits, a, draws, s, what);
}

}  // namespace pldp

using namespace pldp;

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

