"""GPU parity of the fused drafting launch (pldp_draft_step) against the oracle,
over shapes that give one CTA per sequence (both rankings in one CTA) and full
clusters (rankings split across CTAs), and over the degenerate inputs."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from tests._parity import SCORE_TOL, Buffers, check_choice, check_scores, gpu_step, host, snapshot

pytestmark = pytest.mark.gpu
DEV = "cuda"


def i32(x):
    return torch.as_tensor(np.asarray(x, np.int32), device=DEV)


def _compare(g, ids0, L0, H, A, row_idx, agg, ngram, C, K, draft_from, thr=float("-inf"), status0=None):
    """The drafting outputs in g against the oracle on the state (ids0, L0); status0
    (the oracle's bits of an earlier part of the same call) is OR-ed into the status
    expected."""
    o_cand, o_cnt, o_ml, o_st = oracle.find_candidates(ids0, L0, ngram[0], ngram[1], C)
    assert np.array_equal(g["cnt"], o_cnt) and np.array_equal(g["ml"], o_ml)
    for b in range(len(L0)):
        n = min(o_cnt[b], C)
        assert np.array_equal(g["cand"][b, :n], o_cand[b, :n]), b
    st = o_st.copy() if status0 is None else o_st | status0
    valid = np.array([0 <= l <= ids0.shape[1] for l in L0])
    if H is not None:
        o_s, o_b, _ = oracle.rank_hidden(host(H), L0, o_cand, o_cnt, threshold=thr, status=st)
        check_scores(g["scores_h"], o_s, np.where(valid, o_cnt, 0), C)
        check_choice(g["best_h"], o_b, o_s, o_cand, o_cnt, C)
    if A is not None:
        o_s, o_b, _ = oracle.rank_attention(host(A), L0, o_cand, o_cnt, row_idx=row_idx, agg=agg, status=st)
        check_scores(g["scores_a"], o_s, np.where(valid, o_cnt, 0), C)
        if agg == 0:
            assert np.array_equal(g["best_a"], o_b)
        else:
            check_choice(g["best_a"], o_b, o_s, o_cand, o_cnt, C)
    best = g["best_h"] if draft_from == "hidden" else g["best_a"]
    o_d, o_dl = oracle.extract_draft(ids0, L0, best, K)
    assert np.array_equal(g["draft"], o_d) and np.array_equal(g["dlen"], o_dl)
    assert np.array_equal(g["status"].view(np.uint32), st)


# B >= half the SMs with contexts up to 40k tokens take the one-CTA-per-sequence kernel
# (whole context in shared memory); smaller batches take the cluster kernel.
@pytest.mark.parametrize("T,V,B", [(300, 5, 12), (4096, 50, 8), (20000, 7, 3), (36096, 3000, 16),
                                   (3000, 5, 96), (5000, 40, 96), (36096, 3000, 96), (2048, 2, 80)])
@pytest.mark.parametrize("mode", ["both", "hidden", "attention"])
def test_draft_step_random(lib, T, V, B, mode):
    rng = np.random.default_rng(T + V)
    gen = torch.Generator(device=DEV).manual_seed(T)
    C, K, d, R = 64, 10, 256, 12
    ids = rng.integers(0, V, size=(B, T)).astype(np.int32)
    lens = rng.integers(0, T + 1, size=B)
    lens[:3] = [T, 1, 2]
    if B > 4:
        lens[3] = T + 3                       # invalid length
    H = torch.randn((B, T, d), generator=gen, device=DEV).to(torch.bfloat16) if mode != "attention" else None
    A = torch.rand((B, R, T), generator=gen, device=DEV).to(torch.bfloat16) if mode != "hidden" else None
    if A is not None and T % 3 == 0:                  # key-major: the R values of a key side by side
        A = A.transpose(1, 2).contiguous().transpose(1, 2)
    buf = Buffers(B, K, 8, C, DEV)
    draft_from = "attention" if mode == "attention" else "hidden"
    gpu_step(buf, i32(ids), i32(lens), None, H=H, A=A, draft_from=draft_from, append=False, fused=True)
    g = snapshot(buf)
    _compare(g, ids, lens, H, A, None, 0, (1, 3), C, K, draft_from)


@pytest.mark.parametrize("agg", [0, 1])
@pytest.mark.parametrize("layout", ["head", "key"])
def test_draft_step_rows_threshold_long_draft(lib, agg, layout):
    rng = np.random.default_rng(9 + agg)
    B, T, C, K, d, R = 10, 9000, 40, 70, 512, 16
    ids = rng.integers(0, 4, size=(B, T)).astype(np.int32)      # many candidates: overflow
    lens = rng.integers(2, T + 1, size=B)
    H = torch.randn((B, T, d), device=DEV, dtype=torch.float32)
    A = torch.rand((B, R, T), device=DEV, dtype=torch.float32)
    if layout == "key":                                          # the R values of a key side by side
        A = A.transpose(1, 2).contiguous().transpose(1, 2)
    rows = [5, -2, 0, 15, 40, 3]                                  # two invalid rows
    buf = Buffers(B, K, 8, C, DEV)
    gpu_step(buf, i32(ids), i32(lens), None, ngram=(2, 4), H=H, A=A, row_idx=rows, agg=agg,
             threshold=0.02, draft_from="hidden", append=False, fused=True)
    g = snapshot(buf)
    _compare(g, ids, lens, H, A, rows, agg, (2, 4), C, K, "hidden", thr=0.02)


@pytest.mark.parametrize("draft_from", ["hidden", "attention"])
def test_draft_step_matches_separate_calls(lib, draft_from):
    """Same integer results as the four separate calls on a planted workload."""
    w = wl.CONFIGS["attention_b32_ctx8k"].replace(B=24, prompt_len=3000, out_len=1000, V=8000, d=1024, layers=2,
                                 heads=8, planted_heads=2, C_cap=128)
    inp = wl.single_step(w, device=DEV)
    outs = []
    for fused in (False, True):
        buf = Buffers(w.B, w.K, w.V, w.C_cap, DEV)
        gpu_step(buf, inp["ids"], inp["seq_len"], None, H=inp["H"], A=inp["A"], row_idx=inp["row_idx"],
                 draft_from=draft_from, append=False, fused=fused)
        outs.append(snapshot(buf))
    a, b = outs
    for k in ("cand", "cnt", "ml", "best_h", "best_a", "draft", "dlen", "status"):
        assert np.array_equal(a[k], b[k]), k
    np.testing.assert_allclose(a["scores_h"], b["scores_h"], atol=1e-5, equal_nan=True)
    assert np.array_equal(a["scores_a"], b["scores_a"], equal_nan=True)
