"""GPU parity of the rankings on candidate-heavy inputs: contexts from a small
vocabulary with Eq. 1's unigram match, so that x_t has hundreds of earlier
occurrences and every CTA scores many candidates (the warps then stream their
candidates on their own).  The largest case is the benchmark's candidate-heavy
run at its full size (batch 128, context 32768, hidden width 4096, 128 attention
rows); every sequence is compared with the oracle, which is handed host arrays
holding exactly the rows its rankings read."""
import numpy as np
import pytest
import torch

import oracle
from tests._parity import Buffers, check_choice, check_scores, host, oracle_rows, snapshot

pytestmark = pytest.mark.gpu
DEV = "cuda"


# key_major: the R values of a key side by side, as the benchmark holds them.  Under MAX
# with all rows and whole 16-byte runs of a power-of-two count of vectors, Eq. 2 takes
# the dense whole-vector path: 16 vectors a key (R = 128 bf16, R = 64 f32), 4 (R = 32
# bf16) and 128 (R = 1024 bf16, several loads per lane); SUM stays on the value path.
@pytest.mark.parametrize("B,T,V,d,R,dtype,C_cap,thr,agg,key_major", [
    (128, 32768, 64, 4096, 128, torch.bfloat16, 1024, float("-inf"), 0, True),
    (128, 32768, 256, 4096, 128, torch.bfloat16, 1024, float("-inf"), 1, False),
    (24, 9000, 40, 1000, 16, torch.float32, 300, 0.02, 0, False),
    (7, 20000, 30, 768, 48, torch.bfloat16, 2048, float("-inf"), 1, False),
    (16, 6000, 12, 256, 32, torch.bfloat16, 1024, float("-inf"), 0, True),
    (16, 6000, 12, 256, 32, torch.bfloat16, 1024, float("-inf"), 1, True),
    (8, 4000, 8, 128, 1024, torch.bfloat16, 1024, float("-inf"), 0, True),
    (12, 5000, 20, 512, 64, torch.float32, 600, float("-inf"), 0, True),
])
def test_candidate_heavy_rankings(lib, B, T, V, d, R, dtype, C_cap, thr, agg, key_major):
    rng = np.random.default_rng(T + V)
    gen = torch.Generator(device=DEV).manual_seed(V)
    ids = rng.integers(0, V, size=(B, T)).astype(np.int32)
    lens = np.full(B, T, np.int32)
    lens[1] = T // 3                                     # ragged
    lens[2] = 2
    ids_g = torch.as_tensor(ids, device=DEV)
    L_g = torch.as_tensor(lens, device=DEV)
    H = torch.randn((B, T, d), generator=gen, device=DEV).to(dtype)
    A = torch.rand((B, R, T), generator=gen, device=DEV).to(dtype)
    if key_major:
        A = A.transpose(1, 2).contiguous().transpose(1, 2)
    buf = Buffers(B, 8, 8, C_cap, DEV)
    lib.pldp_find_candidates(ids_g, L_g, 1, 1, buf.cand, buf.cnt, buf.ml, buf.status)
    lib.pldp_rank_hidden(H, L_g, buf.cand, buf.cnt, buf.best_h, scores=buf.scores_h, best_score=buf.bscore_h,
                         threshold=thr, status=buf.status)
    lib.pldp_rank_attention(A, L_g, buf.cand, buf.cnt, buf.best_a, agg=agg, scores=buf.scores_a,
                            best_score=buf.bscore_a, status=buf.status)
    g = snapshot(buf)
    o_cand, o_cnt, o_ml, o_st = oracle.find_candidates(ids, lens, 1, 1, C_cap)
    assert np.array_equal(g["cnt"], o_cnt) and np.array_equal(g["ml"], o_ml)
    for b in range(B):
        n = min(o_cnt[b], C_cap)
        assert np.array_equal(g["cand"][b, :n], o_cand[b, :n]), b
    assert np.median(np.minimum(o_cnt, C_cap)) >= min(C_cap, T // V // 2)   # candidate-heavy indeed
    Hs, As = oracle_rows(H, A, lens, o_cand, o_cnt)
    st = o_st.copy()
    o_s, o_b, o_bs = oracle.rank_hidden(Hs, lens, o_cand, o_cnt, threshold=thr, status=st)
    check_scores(g["scores_h"], o_s, o_cnt, C_cap)
    check_choice(g["best_h"], o_b, o_s, o_cand, o_cnt, C_cap)
    o_sa, o_ba, _ = oracle.rank_attention(As, lens, o_cand, o_cnt, agg=agg, status=st)
    check_scores(g["scores_a"], o_sa, o_cnt, C_cap)
    if agg == 0:
        assert np.array_equal(g["best_a"], o_ba)        # the maximum is exact
    else:
        check_choice(g["best_a"], o_ba, o_sa, o_cand, o_cnt, C_cap)
    assert np.array_equal(g["status"].view(np.uint32), st)
