"""GPU parity of every step at oracle-friendly sizes that span several CTAs,
clusters, vector tiles and ragged tails, including the degenerate inputs."""
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


# ----------------------------------------------------------------------------
# candidate search
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("T_cap,V,stride_pad", [(512, 7, 0), (1001, 3, 0), (4096, 40, 4),
                                                (4100, 5000, 0), (20003, 11, 5), (36096, 128256, 0),
                                                (9000, 2, 0)])
@pytest.mark.parametrize("ngram", [(1, 1), (1, 3), (2, 4), (1, 8)])
def test_find_candidates(lib, T_cap, V, stride_pad, ngram):
    rng = np.random.default_rng(T_cap * 7 + V + ngram[1])
    B, C_cap = 24, 300
    ids_full = rng.integers(0, V, size=(B, T_cap + stride_pad)).astype(np.int32)
    # copies of the row tail so that long suffix matches exist
    for b in range(0, B, 3):
        L = rng.integers(3, 10)
        s = rng.integers(0, T_cap // 2)
        ids_full[b, T_cap - 1 - L: T_cap - 1] = ids_full[b, s: s + L]
    lens = rng.integers(0, T_cap + 1, size=B)
    lens[:6] = [0, 1, 2, T_cap, T_cap - 1, 3]
    lens[6] = T_cap + 1          # invalid: flagged
    lens[7] = -4                 # invalid: flagged
    ids_t = i32(ids_full)[:, :T_cap] if stride_pad else i32(ids_full)
    buf = Buffers(B, 4, 8, C_cap, DEV)
    lib.pldp_find_candidates(ids_t, i32(lens), ngram[0], ngram[1], buf.cand, buf.cnt, buf.ml,
                             buf.status, T_cap=T_cap)
    g = snapshot(buf)
    o_cand, o_cnt, o_ml, o_st = oracle.find_candidates(ids_full[:, :T_cap], lens, ngram[0], ngram[1],
                                                       C_cap)
    assert np.array_equal(g["cnt"], o_cnt)
    assert np.array_equal(g["ml"], o_ml)
    assert np.array_equal(g["status"].view(np.uint32), o_st)
    for b in range(B):
        n = min(o_cnt[b], C_cap)
        assert np.array_equal(g["cand"][b, :n], o_cand[b, :n]), b
        assert (g["cand"][b, n:] == -1).all()          # untouched past the list


def test_find_candidates_unaligned_rows(lib):
    """ids not 16-byte aligned (scalar path)."""
    rng = np.random.default_rng(5)
    B, T = 9, 3001
    base = i32(rng.integers(0, 5, size=B * T + 1))
    ids = base[1:].view(B, T)
    lens = rng.integers(0, T + 1, size=B)
    buf = Buffers(B, 4, 8, 64, DEV)
    lib.pldp_find_candidates(ids, i32(lens), 1, 3, buf.cand, buf.cnt, buf.ml, buf.status)
    g = snapshot(buf)
    o_cand, o_cnt, o_ml, o_st = oracle.find_candidates(host(ids), lens, 1, 3, 64)
    assert np.array_equal(g["cnt"], o_cnt) and np.array_equal(g["ml"], o_ml)
    for b in range(B):
        n = min(o_cnt[b], 64)
        assert np.array_equal(g["cand"][b, :n], o_cand[b, :n])


def test_find_candidates_zero_capacity(lib):
    ids = i32(np.tile(np.arange(6) % 2, (3, 1)))
    buf = Buffers(3, 4, 8, 1, DEV)
    cand = torch.zeros((3, 0), dtype=torch.int32, device=DEV)
    lib.pldp_find_candidates(ids, i32([6, 6, 1]), 1, 3, cand, buf.cnt, buf.ml, buf.status)
    g = snapshot(buf)
    _, o_cnt, o_ml, o_st = oracle.find_candidates(host(ids), [6, 6, 1], 1, 3, 0)
    assert np.array_equal(g["cnt"], o_cnt) and np.array_equal(g["status"].view(np.uint32), o_st)


# ----------------------------------------------------------------------------
# hidden ranking
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("d,dtype", [(64, torch.bfloat16), (4096, torch.bfloat16),
                                     (5120, torch.bfloat16), (257, torch.float32),
                                     (4096, torch.float32), (100, torch.bfloat16), (3, torch.float32)])
@pytest.mark.parametrize("C_cap", [8, 200])
def test_rank_hidden(lib, d, dtype, C_cap):
    rng = np.random.default_rng(d + C_cap)
    gen = torch.Generator(device=DEV).manual_seed(d)
    B, T = 12, 300
    H = torch.randn((B, T, d), generator=gen, device=DEV).to(dtype)
    lens = rng.integers(0, T + 1, size=B)
    lens[:4] = [0, 1, 2, 3]
    lens[4] = T + 5                              # invalid
    cands = np.stack([np.sort(rng.choice(T, C_cap, replace=False)) for _ in range(B)]).astype(np.int32)
    cands[:, 0] = 0                              # j = 0 is never eligible
    cnt = rng.integers(0, C_cap + 40, size=B)   # beyond C_cap: clipped to the list
    cnt[5] = -3
    for b in range(6, B):                        # planted near-copies and exact ties
        t = lens[b] - 1
        if t >= 3 and C_cap > 1:
            j = cands[b, 1]
            if 1 <= j < t:
                H[b, j - 1] = H[b, t - 1] * 2
    buf = Buffers(B, 4, 8, C_cap, DEV)
    thr = float("-inf") if C_cap == 8 else 0.01
    lib.pldp_rank_hidden(H, i32(lens), i32(cands), i32(cnt), buf.best_h, scores=buf.scores_h,
                         best_score=buf.bscore_h, threshold=thr, status=buf.status)
    g = snapshot(buf)
    st = np.zeros(B, np.uint32)
    o_s, o_b, o_bs = oracle.rank_hidden(host(H), lens, cands, cnt, threshold=thr, status=st)
    assert np.array_equal(g["status"].view(np.uint32), st)
    ok = np.array([0 <= l <= T for l in lens])
    check_scores(g["scores_h"], o_s, np.where(ok, cnt, 0), C_cap)
    check_choice(g["best_h"], o_b, o_s, cands, cnt, C_cap)
    fin = g["best_h"] >= 0
    assert np.all(np.abs(g["bscore_h"][fin] - o_bs[fin]) <= SCORE_TOL)
    assert np.all(np.isneginf(g["bscore_h"][~fin]))


def test_rank_hidden_tie_goes_to_smaller_position(lib):
    B, T, d = 4, 64, 4096
    H = torch.randn((B, T, d), device=DEV).to(torch.bfloat16)
    t = T - 1
    for b in range(B):
        H[b, 10] = H[b, t - 1]
        H[b, 40] = H[b, t - 1]
    cands = np.tile(np.array([41, 11, 30, 50], np.int32), (B, 1))
    buf = Buffers(B, 4, 8, 4, DEV)
    lib.pldp_rank_hidden(H, i32([T] * B), i32(cands), i32([4] * B), buf.best_h)
    assert snapshot(buf)["best_h"].tolist() == [11] * B


# ----------------------------------------------------------------------------
# attention ranking
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("agg", [0, 1])
@pytest.mark.parametrize("rows", [None, [3, 0, 7, 15], [2, -1, 99, 5]])
@pytest.mark.parametrize("layout", ["head", "key"])
def test_rank_attention(lib, dtype, agg, rows, layout):
    rng = np.random.default_rng(3 + agg)
    B, R, T, C_cap = 10, 16, 777, 96
    A = torch.rand((B, R, T), device=DEV).to(dtype)
    if layout == "key":                                  # the same values, the R of a key side by side
        A = A.transpose(1, 2).contiguous().transpose(1, 2)
    A[:, :, 5] = A[:, :, 9]                           # ties between columns 5 and 9
    lens = rng.integers(0, T + 1, size=B)
    lens[:3] = [0, 1, T]
    cands = np.stack([np.sort(rng.choice(T, C_cap, replace=False)) for _ in range(B)]).astype(np.int32)
    cands[:, :2] = [5, 9]
    cnt = rng.integers(0, C_cap + 1, size=B)
    buf = Buffers(B, 4, 8, C_cap, DEV)
    lib.pldp_rank_attention(A, i32(lens), i32(cands), i32(cnt), buf.best_a, row_idx=None if rows is None
                            else i32(rows), agg=agg, scores=buf.scores_a, best_score=buf.bscore_a,
                            status=buf.status)
    g = snapshot(buf)
    st = np.zeros(B, np.uint32)
    o_s, o_b, o_bs = oracle.rank_attention(host(A), lens, cands, cnt, row_idx=rows, agg=agg, status=st)
    assert np.array_equal(g["status"].view(np.uint32), st)
    check_scores(g["scores_a"], o_s, cnt, C_cap)
    if agg == 0:
        assert np.array_equal(g["best_a"], o_b)        # max is exact
    else:
        check_choice(g["best_a"], o_b, o_s, cands, cnt, C_cap)


# ----------------------------------------------------------------------------
# draft
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("K", [1, 10, 70])
def test_extract_draft(lib, K):
    rng = np.random.default_rng(K)
    B, T = 50, 200
    ids = rng.integers(0, 1000, size=(B, T)).astype(np.int32)
    lens = rng.integers(-2, T + 3, size=B)
    best = rng.integers(-2, T + 2, size=B)
    buf = Buffers(B, K, 8, 4, DEV)
    lib.pldp_extract_draft(i32(ids), i32(lens), i32(best), buf.draft, buf.dlen)
    g = snapshot(buf)
    o_d, o_l = oracle.extract_draft(ids, lens, best, K)
    assert np.array_equal(g["draft"], o_d) and np.array_equal(g["dlen"], o_l)


# ----------------------------------------------------------------------------
# verification
# ----------------------------------------------------------------------------
# V * sizeof(dtype): >= 2 KB and a multiple of 16 bytes takes the streaming path (32000,
# 1000 f32, 128256); a multiple of 16 bytes under 2 KB takes the short-row path (1000 and
# 64 bf16); anything else takes element loads (1001, 999, 7).
@pytest.mark.parametrize("V,dtype", [(32000, torch.bfloat16), (1000, torch.float32),
                                     (1001, torch.bfloat16), (999, torch.float32), (7, torch.bfloat16),
                                     (128256, torch.bfloat16), (1000, torch.bfloat16), (64, torch.bfloat16)])
@pytest.mark.parametrize("K", [1, 10, 40])
def test_verify_greedy(lib, V, dtype, K):
    rng = np.random.default_rng(V + K)
    B, T_cap = 9, 64
    gen = torch.Generator(device=DEV).manual_seed(V * K)
    logits = torch.randn((B, K + 1, V), generator=gen, device=DEV)
    logits = (logits * 2).round().to(dtype)            # many exact ties at the max
    logits[0, 0] = 0.0
    logits[0, 0, 3:] = -0.0                            # -0.0 and +0.0 tie: index 0 wins
    am = host(logits.float()).argmax(-1)
    draft = np.where(rng.random((B, K)) < 0.85, am[:, :K], rng.integers(-3, V + 3, size=(B, K)))
    dlen = rng.integers(0, K + 1, size=B)
    dlen[1], dlen[2] = K + 4, -1                       # clamped, flagged
    ids = rng.integers(0, V, size=(B, T_cap)).astype(np.int32)
    lens = rng.integers(1, T_cap - K - 1, size=B)
    lens[3] = T_cap - 1                                # capacity overflow
    lens[4] = 0                                        # invalid
    ids_g, lens_g = i32(ids), i32(lens)
    buf = Buffers(B, K, V, 4, DEV)
    for rep in range(2):                               # the workspace resets itself
        ids_g.copy_(i32(ids))
        lens_g.copy_(i32(lens))
        buf.status.zero_()
        lib.pldp_verify_greedy(logits, i32(draft), i32(dlen), buf.acc, buf.nxt, buf.ws, argmax=buf.argmax,
                               ids=ids_g, seq_len=lens_g, kv_keep_len=buf.kv, status=buf.status)
        g = snapshot(buf)
        ids_o, lens_o = ids.copy(), lens.astype(np.int32).copy()
        o = oracle.verify_greedy(host(logits), draft, dlen, ids=ids_o, seq_len=lens_o, kv_keep=True)
        assert np.array_equal(g["argmax"], o["argmax"])
        assert np.array_equal(g["acc"], o["accept_len"])
        assert np.array_equal(g["nxt"], o["next_token"])
        assert np.array_equal(g["kv"], o["kv_keep_len"])
        assert np.array_equal(g["status"].view(np.uint32), o["status"])
        assert np.array_equal(host(ids_g), ids_o) and np.array_equal(host(lens_g), lens_o)
        assert int(buf.ws.count_nonzero()) == 0


def test_verify_without_bookkeeping_and_large_batch(lib):
    B, K, V = 300, 3, 4096
    logits = torch.randn((B, K + 1, V), device=DEV, dtype=torch.bfloat16)
    draft = torch.randint(0, V, (B, K), device=DEV, dtype=torch.int32)
    dlen = torch.full((B,), K, device=DEV, dtype=torch.int32)
    buf = Buffers(B, K, V, 4, DEV)
    lib.pldp_verify_greedy(logits, draft, dlen, buf.acc, buf.nxt, buf.ws, argmax=buf.argmax)
    g = snapshot(buf)
    o = oracle.verify_greedy(host(logits), host(draft), host(dlen))
    assert np.array_equal(g["argmax"], o["argmax"]) and np.array_equal(g["acc"], o["accept_len"])
    assert np.array_equal(g["nxt"], o["next_token"])


# ----------------------------------------------------------------------------
# a whole step on a small synthetic workload, both rankings
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("draft_from", ["hidden", "attention"])
def test_small_step_end_to_end(lib, draft_from):
    w = wl.CONFIGS["attention_b32_ctx8k"].replace(B=6, prompt_len=900, out_len=300, V=3000, d=512, layers=2,
                                 heads=8, planted_heads=2, C_cap=128)
    inp = wl.single_step(w, device=DEV)
    ids0, L0 = host(inp["ids"]), host(inp["seq_len"])
    buf = Buffers(w.B, w.K, w.V, w.C_cap, DEV)
    gpu_step(buf, inp["ids"], inp["seq_len"], inp["logits"], H=inp["H"], A=inp["A"],
             row_idx=inp["row_idx"], draft_from=draft_from)
    g = snapshot(buf)
    o_cand, o_cnt, o_ml, _ = oracle.find_candidates(ids0, L0, 1, 3, w.C_cap)
    assert np.array_equal(g["cnt"], o_cnt) and np.array_equal(g["ml"], o_ml)
    o_sh, o_bh, _ = oracle.rank_hidden(host(inp["H"]), L0, o_cand, o_cnt)
    o_sa, o_ba, _ = oracle.rank_attention(host(inp["A"]), L0, o_cand, o_cnt, row_idx=inp["row_idx"])
    check_scores(g["scores_h"], o_sh, o_cnt, w.C_cap)
    check_scores(g["scores_a"], o_sa, o_cnt, w.C_cap)
    check_choice(g["best_h"], o_bh, o_sh, o_cand, o_cnt, w.C_cap)
    assert np.array_equal(g["best_a"], o_ba)
    best = g["best_h"] if draft_from == "hidden" else g["best_a"]
    o_d, o_dl = oracle.extract_draft(ids0, L0, best, w.K)
    assert np.array_equal(g["draft"], o_d)
    ids_o, L_o = ids0.copy(), L0.copy()
    o = oracle.verify_greedy(host(inp["logits"]), o_d, o_dl, ids=ids_o, seq_len=L_o)
    assert np.array_equal(g["acc"], o["accept_len"]) and np.array_equal(g["nxt"], o["next_token"])
    assert np.array_equal(host(inp["ids"]), ids_o) and np.array_equal(host(inp["seq_len"]), L_o)
    # the planted source is found and the planted accept length reproduced
    assert np.array_equal(g["acc"], inp["planted_accept"])
