"""GPU parity of the ranking variants of App. B against the oracle: the averaged
hidden-state ranking (pldp_rank_hidden_avg, App. B.2).  The threshold (App. B.3)
and SUM aggregation are covered with the main calls."""
import numpy as np
import pytest
import torch

import oracle
from tests._parity import SCORE_TOL, Buffers, check_choice, check_scores, host, snapshot

pytestmark = pytest.mark.gpu
DEV = "cuda"


def i32(x):
    return torch.as_tensor(np.asarray(x, np.int32), device=DEV)


# d * sizeof: 16-byte rows take vector loads (64 and 4096 bf16, 100 f32); others element loads
@pytest.mark.parametrize("d,dtype", [(64, torch.bfloat16), (4096, torch.bfloat16), (100, torch.float32),
                                     (99, torch.float32), (1001, torch.bfloat16)])
@pytest.mark.parametrize("m", [1, 2, 5])
@pytest.mark.parametrize("C_cap", [8, 200])
def test_rank_hidden_avg(lib, d, dtype, m, C_cap):
    rng = np.random.default_rng(d + m + C_cap)
    gen = torch.Generator(device=DEV).manual_seed(d * m)
    B, T = 12, 300
    H = torch.randn((B, T, d), generator=gen, device=DEV).to(dtype)
    lens = rng.integers(0, T + 1, size=B)
    lens[:4] = [0, 1, 2, 3]
    lens[4] = T + 5                              # invalid
    cands = np.stack([np.sort(rng.choice(T, C_cap, replace=False)) for _ in range(B)]).astype(np.int32)
    cands[:, 0] = 0                              # never eligible
    cands[6, 1] = 1                              # window cut at position 0
    cnt = rng.integers(0, C_cap + 40, size=B)
    cnt[5] = -3
    for b in range(7, B):                        # planted near-copies of the query window
        t = lens[b] - 1
        if t >= m + 2 and C_cap > 1:
            j = cands[b, 1]
            if m <= j < t:
                H[b, j - m:j] = H[b, t - m:t] * 2
    buf = Buffers(B, 4, 8, C_cap, DEV)
    thr = float("-inf") if C_cap == 8 else 0.01
    lib.pldp_rank_hidden_avg(H, i32(lens), i32(cands), i32(cnt), buf.best_h, m, scores=buf.scores_h,
                             best_score=buf.bscore_h, threshold=thr, status=buf.status)
    g = snapshot(buf)
    st = np.zeros(B, np.uint32)
    o_s, o_b, o_bs = oracle.rank_hidden_avg(host(H), lens, cands, cnt, m, threshold=thr, status=st)
    assert np.array_equal(g["status"].view(np.uint32), st)
    ok = np.array([0 <= l <= T for l in lens])
    check_scores(g["scores_h"], o_s, np.where(ok, cnt, 0), C_cap)
    check_choice(g["best_h"], o_b, o_s, cands, cnt, C_cap)
    fin = g["best_h"] >= 0
    assert np.all(np.abs(g["bscore_h"][fin] - o_bs[fin]) <= SCORE_TOL)
    assert np.all(np.isneginf(g["bscore_h"][~fin]))


def test_rank_hidden_avg_m1_agrees_with_eq3(lib):
    rng = np.random.default_rng(5)
    B, T, d, C = 16, 2000, 512, 32
    H = torch.randn((B, T, d), device=DEV, dtype=torch.bfloat16)
    lens = rng.integers(T // 2, T + 1, size=B).astype(np.int32)
    cands = np.stack([np.sort(rng.choice(T // 2, C, replace=False)) for _ in range(B)]).astype(np.int32)
    cnt = np.full(B, C, np.int32)
    outs = []
    for avg in (False, True):
        buf = Buffers(B, 4, 8, C, DEV)
        if avg:
            lib.pldp_rank_hidden_avg(H, i32(lens), i32(cands), i32(cnt), buf.best_h, 1, scores=buf.scores_h)
        else:
            lib.pldp_rank_hidden(H, i32(lens), i32(cands), i32(cnt), buf.best_h, scores=buf.scores_h)
        outs.append(snapshot(buf))
    assert np.array_equal(outs[0]["best_h"], outs[1]["best_h"])
    np.testing.assert_allclose(outs[0]["scores_h"], outs[1]["scores_h"], atol=1e-5, equal_nan=True)
