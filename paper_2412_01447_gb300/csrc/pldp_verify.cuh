// Verification pieces shared by pldp_verify_greedy (verify.cu), pldp_verify_sample
// (sample.cu) and the fused verification + next draft calls (draft_step.cu): the
// argument block, the per-sequence finish (accept, bonus, append; Sec. 4.4), the
// launch of the streaming argmax pass and that of the sampling draws.
#pragma once

#include "pldp_internal.cuh"

namespace pldp {

struct VerifyArgs {
    const int32_t* draft;
    const int32_t* draft_len;
    int32_t* argmax;
    int32_t* accept_len;
    int32_t* next_token;
    int32_t* ids;
    int64_t ids_stride;
    int32_t* seq_len;
    int64_t T_cap;
    int32_t* kv_keep_len;
    uint32_t* status;
    unsigned long long* row_keys;   // [B*(K+1)], zero between calls (greedy)
    const int32_t* row_draws;       // [B*(K+1)] the draws of sampling verification, or null (greedy)
    int B, K, V;
};

// Where the finish reads the K+1 target tokens of a sequence: the greedy row keys
// (argmax packed in the low word; the keys are returned to zero afterwards), the
// draws of sampling verification staged in shared memory, or either (RowTokens).
struct KeyTokens {
    unsigned long long* keys;   // [K+1] of this sequence
    __device__ __forceinline__ int at(int i) const { return static_cast<int>(key_index(__ldcg(keys + i))); }
    __device__ __forceinline__ void release(int K1, int lane) const {
        for (int i = lane; i < K1; i += 32) keys[i] = 0ull;
    }
};
struct SharedTokens {
    const int32_t* tok;          // shared memory, [K+1]
    __device__ __forceinline__ int at(int i) const { return tok[i]; }
    __device__ __forceinline__ void release(int, int) const {}
};

// Either of the two, chosen per call: the draws when they are given (written by
// the previous kernel, read through L2), else the greedy row keys.
struct RowTokens {
    unsigned long long* keys;    // [K+1] of this sequence (greedy)
    const int32_t* draws;        // [K+1] of this sequence (sampling), or null
    __device__ __forceinline__ int at(int i) const {
        return draws ? __ldcg(draws + i) : static_cast<int>(key_index(__ldcg(keys + i)));
    }
    __device__ __forceinline__ void release(int K1, int lane) const {
        if (!draws)
            for (int i = lane; i < K1; i += 32) keys[i] = 0ull;
    }
};

// What the finish decided, for a caller that continues with the extended context.
struct FinishOut {
    int n;          // accepted draft tokens
    int bonus;      // the token emitted after them
    bool appended;  // draft[0..n-1] and bonus were written at positions L .. L+n
};

// The finish's inputs that do not depend on the target tokens (the draft length,
// the context length and lane i's draft token i), for a caller that reads them
// before the tokens are final.
struct FinishIn {
    int d_in;
    int64_t L;
    int tok_first;
};

__device__ __forceinline__ FinishIn finish_inputs(const VerifyArgs& a, int64_t b, int lane) {
    return FinishIn{a.draft_len[b], a.seq_len ? static_cast<int64_t>(a.seq_len[b]) : 0,
                    lane < a.K ? a.draft[b * a.K + lane] : 0};
}

// Accept/bonus/append for sequence b, by one warp, once its K+1 target tokens are
// final.  Everything it reads is requested up front (one round trip when K < 32);
// `in` (optional) holds the inputs that were read earlier.
// Sec. 4.4: n = first i < d with draft_i != target_i (else d), bonus = target_n.
// Returns (in every lane) the context length after the call: L + n + 1 when the
// tokens were appended, L when they were not (capacity, no ids), -1 when seq_len
// is absent or out of range.
template <typename Src>
__device__ int64_t finish_sequence(const VerifyArgs& a, int64_t b, int lane, const Src& src,
                                   FinishOut* out = nullptr, const FinishIn* in = nullptr) {
    const int K1 = a.K + 1;
    const FinishIn fi = in ? *in : finish_inputs(a, b, lane);
    const int d_in = fi.d_in;
    const int64_t L = fi.L;
    const int t_first = lane < K1 ? src.at(lane) : 0;
    const int tok_first = fi.tok_first;
    uint32_t st = 0;
    int d = d_in;
    if (d < 0 || d > a.K) {
        st |= PLDP_ST_DRAFT_LEN;
        d = d < 0 ? 0 : a.K;
    }
    int n = d;
    bool range_bad = false;
    for (int i0 = 0; i0 < K1; i0 += 32) {
        const int i = i0 + lane;
        const int am = i0 == 0 ? t_first : (i < K1 ? src.at(i) : 0);
        const int tok = i0 == 0 ? tok_first : (i < a.K ? a.draft[b * a.K + i] : 0);
        if (i < K1 && a.argmax) a.argmax[b * K1 + i] = am;
        const bool in_draft = i < d;
        range_bad |= in_draft && (tok < 0 || tok >= a.V);
        const unsigned mism = __ballot_sync(0xFFFFFFFFu, in_draft && tok != am);
        if (n == d && mism) n = i0 + __ffs(mism) - 1;
    }
    if (__any_sync(0xFFFFFFFFu, range_bad)) st |= PLDP_ST_TOKEN_RANGE;
    const int bonus = n < 32 ? __shfl_sync(0xFFFFFFFFu, t_first, n) : src.at(n);
    __syncwarp();
    src.release(K1, lane);

    if (lane == 0) {
        a.accept_len[b] = n;
        a.next_token[b] = bonus;
    }
    int64_t L_after = -1;
    if (a.seq_len) {
        int64_t kv = -1;
        if (L < 1 || L > a.T_cap) {
            st |= PLDP_ST_SEQ_LEN;
        } else {
            kv = L + n;
            L_after = L;
            if (L + n + 1 > a.T_cap) {
                st |= PLDP_ST_CAPACITY;
            } else {
                if (a.ids) {
                    int32_t* row = a.ids + b * a.ids_stride + L;
                    if (lane < n) row[lane] = tok_first;
                    for (int i = 32 + lane; i < n; i += 32) row[i] = a.draft[b * a.K + i];
                    if (lane == 0) row[n] = bonus;
                }
                __syncwarp();
                if (lane == 0) a.seq_len[b] = static_cast<int32_t>(L + n + 1);
                L_after = L + n + 1;
            }
        }
        if (a.kv_keep_len && lane == 0) a.kv_keep_len[b] = static_cast<int32_t>(kv);
    }
    if (lane == 0) {
        if (a.status && st) a.status[b] |= st;
    }
    if (out) {
        out->n = n;
        out->bonus = bonus;
        out->appended = a.seq_len && a.ids && L_after == L + n + 1;
    }
    return L_after;
}

// The argument block of pldp_verify_greedy (row_keys left unset).
VerifyArgs verify_args(int B, int K, int V, const int32_t* draft, const int32_t* draft_len,
                       int32_t* argmax, int32_t* accept_len, int32_t* next_token, int32_t* ids,
                       int64_t ids_stride, int32_t* seq_len, int64_t T_cap, int32_t* kv_keep_len,
                       uint32_t* status);

// Sampling verification's draws for the fused sampling + next draft call: launches
// the stats pass and one warp per row that draws (Sec. 4.4 at temperature T, from
// the caller's uniforms), leaving the draws in the workspace and setting
// a.row_draws.  The workspace holds the per-piece stats, then the draws
// (sample_draft_workspace_size bytes, 16-byte aligned, no zeroing needed).
size_t sample_draft_workspace_size(int B, int K, int V, pldp_dtype dtype);
pldp_status launch_sample_draws(const void* logits, pldp_dtype dtype, VerifyArgs& a, float temperature,
                                const float* uniforms, void* workspace, cudaStream_t s, const char* what);

// Launches the streaming argmax pass over logits [B, K+1, V] that leaves each
// row's key in `scratch` (pldp_verify_workspace_size bytes, zero between calls)
// and sets a.row_keys.  The caller launches the finish after it, with
// programmatic dependent launch.
pldp_status launch_verify_pass(const void* logits, pldp_dtype dtype, VerifyArgs& a, void* scratch,
                               cudaStream_t s, const char* what);

}  // namespace pldp
