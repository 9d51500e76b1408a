"""The incremental token index of pldp_draft_step: every output must equal the
scanning step's bit for bit (same candidates, counts, match lengths, scores,
choices, drafts, status), and the oracle's at every step, over random contexts,
a decode loop with greedy appends, long appends, shrunk and empty contexts and
tokens the index cannot hold."""
import numpy as np
import pytest
import torch

import oracle
import paper_2412_01447_gb300 as pk
import workloads as wl
from tests._parity import Buffers, gpu_step, host, snapshot
from tests.test_gpu_fused import _compare

pytestmark = pytest.mark.gpu
DEV = "cuda"


def i32(x):
    return torch.as_tensor(np.asarray(x, np.int32), device=DEV)


def _draft(buf, ids, L, K, H=None, A=None, index=None, V=None, ngram=(1, 3), draft_from="hidden"):
    buf.status.zero_()
    pk.pldp_draft_step(ids, L, ngram[0], ngram[1], buf.cand, buf.cnt, buf.ml, K, buf.draft, buf.dlen,
                       None if index is not None else buf.dws, H=H, best_h=buf.best_h if H is not None else None,
                       h_scores=buf.scores_h, best_h_score=buf.bscore_h, A=A,
                       best_a=buf.best_a if A is not None else None, a_scores=buf.scores_a,
                       best_a_score=buf.bscore_a, draft_from=draft_from, status=buf.status, index=index, V=V)
    return snapshot(buf)


DRAFT_OUT = ("cand", "cnt", "ml", "status", "best_h", "best_a", "scores_h", "scores_a", "bscore_h", "bscore_a",
             "draft", "dlen")


def _same(a, b):
    for k in DRAFT_OUT:
        assert np.array_equal(a[k], b[k], equal_nan=True), k


def _ilen(index, B):
    return host(index[:4 * B].view(torch.int32))


# V sets how many occurrences x_t has: hundreds (scanned), 9..15 (suffix matches first,
# then the candidates scored), up to 8 (all scored in one pass)
@pytest.mark.parametrize("T,V,B", [(300, 4, 12), (4096, 50, 8), (4096, 300, 8), (8000, 3000, 16), (2048, 2, 20)])
@pytest.mark.parametrize("mode", ["both", "hidden", "attention"])
def test_indexed_step_equals_scan(lib, T, V, B, mode):
    _indexed_case(T, V, B, mode, C=64, K=10, ngram=(1, 3))


@pytest.mark.parametrize("T,V,B", [(4096, 50, 8), (4096, 300, 8), (8000, 3000, 16), (30000, 20000, 6)])
@pytest.mark.parametrize("C,K,ngram", [(2, 70, (1, 3)), (1, 5, (2, 4)), (3, 64, (1, 8))])
def test_indexed_step_small_caps(lib, T, V, B, C, K, ngram):
    """Candidate lists shorter than the occurrences scored in one pass, drafts longer
    than the staged window, and other n-gram ranges."""
    _indexed_case(T, V, B, "both", C=C, K=K, ngram=ngram)


def _indexed_case(T, V, B, mode, C, K, ngram):
    rng = np.random.default_rng(T + V)
    gen = torch.Generator(device=DEV).manual_seed(T + 1)
    d, R = 128, 12
    T_cap = T + 2000
    ids = rng.integers(0, V, size=(B, T_cap)).astype(np.int32)
    lens = rng.integers(0, T + 1, size=B)
    lens[:3] = [T, 1, 2]
    lens[3] = T_cap + 3                                              # invalid length
    if B > 6:
        lens[6] = 0                                                  # empty, then grows
    H = torch.randn((B, T_cap, d), generator=gen, device=DEV).to(torch.bfloat16) if mode != "attention" else None
    A = torch.rand((B, R, T_cap), generator=gen, device=DEV).to(torch.bfloat16) if mode != "hidden" else None
    draft_from = "attention" if mode == "attention" else "hidden"
    ids_g, L_g = i32(ids), i32(lens)
    index = torch.empty(pk.pldp_index_size(B, V), dtype=torch.uint8, device=DEV)
    st = torch.zeros(B, dtype=torch.int32, device=DEV)
    pk.pldp_index_build(ids_g, L_g, V, index, status=st)
    assert host(st)[3] == pk.PLDP_ST_SEQ_LEN and (np.delete(host(st), 3) == 0).all()
    a, b_ = Buffers(B, K, 8, C, DEV), Buffers(B, K, 8, C, DEV)
    for step in range(5):
        g_scan = _draft(a, ids_g, L_g, K, H, A, ngram=ngram, draft_from=draft_from)
        g_idx = _draft(b_, ids_g, L_g, K, H, A, index=index, V=V, ngram=ngram, draft_from=draft_from)
        _same(g_scan, g_idx)
        _compare(g_idx, ids, lens, H, A, None, 0, ngram, C, K, draft_from)     # every step against the oracle
        # the contexts grow: 1..13 tokens, one long append, one sequence cut back
        L = host(L_g).astype(np.int64)
        for s in range(B):
            if not (0 <= L[s] <= T_cap):
                continue
            n = 600 if (step == 1 and s == 4) else int(rng.integers(1, 14))
            n = min(n, T_cap - L[s])
            ids[s, L[s]:L[s] + n] = rng.integers(0, V, size=n)
            L[s] += n
        if step == 2:
            L[5] = max(L[5] // 2, 1)                                 # shrunk: the index of 5 is unusable
        lens = L.astype(np.int32)
        ids_g.copy_(i32(ids))
        L_g.copy_(i32(lens))
    il = _ilen(index, B)
    assert il[3] == -1 and il[5] == -1
    if B > 6:
        assert il[6] >= 0                                            # the context that was empty kept its index


def test_index_marks_tokens_it_cannot_hold(lib):
    B, T, V = 4, 500, 100
    rng = np.random.default_rng(1)
    ids = rng.integers(0, V, size=(B, T)).astype(np.int32)
    ids[2, 17] = V + 5
    lens = np.full(B, T - 50, np.int32)
    ids_g, L_g = i32(ids), i32(lens)
    index = torch.empty(pk.pldp_index_size(B, V), dtype=torch.uint8, device=DEV)
    st = torch.zeros(B, dtype=torch.int32, device=DEV)
    pk.pldp_index_build(ids_g, L_g, V, index, status=st)
    assert host(st).tolist() == [0, 0, pk.PLDP_ST_TOKEN_RANGE, 0]
    assert _ilen(index, B).tolist() == [T - 51, T - 51, -1, T - 51]
    H = torch.randn((B, T, 64), device=DEV, dtype=torch.bfloat16)
    a, b_ = Buffers(B, 8, 8, 32, DEV), Buffers(B, 8, 8, 32, DEV)
    _same(_draft(a, ids_g, L_g, 8, H), _draft(b_, ids_g, L_g, 8, H, index=index, V=V))


def test_indexed_decode_loop(lib):
    """A sustained loop (batch 32, context 4096, V 128256): each step drafts with and
    without the index on the same state, then verifies greedily with append."""
    w = wl.CONFIGS["decode_loop_b128_ctx32k"].replace(B=32, prompt_len=3072, out_len=1024, d=512)
    steps = 6
    loop = wl.DecodeLoop(w, steps=steps, device=DEV)
    B, K, C = w.B, w.K, w.C_cap
    index = torch.empty(pk.pldp_index_size(B, w.V), dtype=torch.uint8, device=DEV)
    pk.pldp_index_build(loop.ids, loop.seq_len, w.V, index)
    a, b_ = Buffers(B, K, w.V, C, DEV), Buffers(B, K, w.V, C, DEV)
    for s in range(steps):
        loop.step_inputs(s)
        ids0, L0 = host(loop.ids), host(loop.seq_len)
        g_idx = _draft(b_, loop.ids, loop.seq_len, K, loop.H, loop.A, index=index, V=w.V)
        _same(_draft(a, loop.ids, loop.seq_len, K, loop.H, loop.A), g_idx)
        _compare(g_idx, ids0, L0, loop.H, loop.A, None, 0, (w.ngram_min, w.ngram_max), C, K, "hidden")
        pk.pldp_verify_greedy(loop.logits, b_.draft, b_.dlen, b_.acc, b_.nxt, b_.ws, ids=loop.ids,
                              seq_len=loop.seq_len, kv_keep_len=b_.kv, status=b_.status)
        o = oracle.verify_greedy(host(loop.logits), g_idx["draft"], g_idx["dlen"], ids=ids0, seq_len=L0)
        assert np.array_equal(host(b_.acc), o["accept_len"]) and np.array_equal(host(b_.nxt), o["next_token"])
        assert np.array_equal(host(loop.ids), ids0) and np.array_equal(host(loop.seq_len), L0)
    torch.cuda.synchronize()
    L = host(loop.seq_len)
    il = _ilen(index, B)
    assert (il >= 0).all() and (il < L).all()                    # usable, and behind the context
    ids, gt = host(loop.ids), loop.gt_host
    for b in range(B):
        assert np.array_equal(ids[b, :L[b]], gt[b, :L[b]]), b
