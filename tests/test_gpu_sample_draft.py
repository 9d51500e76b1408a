"""pldp_verify_sample_draft (sampling verification of a step, then the next step's
drafting with the token index, in one call) against pldp_verify_sample followed by
pldp_draft_step on the same state -- every output, the extended contexts and the
index bit for bit, step after step -- and against the oracle: the draws as in
the sampling tests (equal, or the uniform within rounding of a boundary of the
exact cumulative distribution), the acceptance, bonus and append following from
the GPU's draws exactly, and the next draft equal to the oracle's on the state
that verification leaves."""
import numpy as np
import pytest
import torch

import oracle
import paper_2412_01447_gb300 as pk
import workloads as wl
from tests._parity import Buffers, host
from tests.test_gpu_fused import _compare
from tests.test_gpu_sample import _f64, _valid_draw
from tests.test_gpu_verify_draft import _draft, _same, _same_index, _snap

pytestmark = pytest.mark.gpu
DEV = "cuda"


def i32(x):
    return torch.as_tensor(np.asarray(x, np.int32), device=DEV)


def _kw(buf, H, A, draft_from):
    return dict(H=H, best_h=buf.best_h if H is not None else None, h_scores=buf.scores_h,
                best_h_score=buf.bscore_h, A=A, best_a=buf.best_a if A is not None else None,
                a_scores=buf.scores_a, best_a_score=buf.bscore_a, draft_from=draft_from, status=buf.status)


def _separate(buf, logits, u, T, ids, L, index, V, H, A, ngram, draft_from):
    B, K1, _ = logits.shape
    ws = torch.empty(pk.pldp_verify_sample_workspace_size(B, K1 - 1, V, logits.dtype), dtype=torch.uint8, device=DEV)
    pk.pldp_verify_sample(logits, u, buf.draft, buf.dlen, buf.acc, buf.nxt, ws, temperature=T, sampled=buf.argmax,
                          ids=ids, seq_len=L, kv_keep_len=buf.kv, status=buf.status)
    _draft(buf, ids, L, index, V, H, A, ngram, draft_from)


def _fused(buf, logits, u, T, ids, L, index, V, H, A, ngram, draft_from, shared=True):
    B, K1, _ = logits.shape
    ws = torch.empty(pk.pldp_verify_sample_draft_workspace_size(B, K1 - 1, V, logits.dtype), dtype=torch.uint8,
                     device=DEV)
    if shared:
        nd, nl = buf.draft, buf.dlen
    else:
        nd, nl = torch.full_like(buf.draft, -7), torch.full_like(buf.dlen, -7)
    pk.pldp_verify_sample_draft(logits, u, buf.draft, buf.dlen, buf.acc, buf.nxt, ws, ids, L, ngram[0], ngram[1],
                                buf.cand, buf.cnt, buf.ml, nd, nl, index, temperature=T, sampled=buf.argmax,
                                kv_keep_len=buf.kv, **_kw(buf, H, A, draft_from))
    if not shared:
        buf.draft.copy_(nd)
        buf.dlen.copy_(nl)


def _oracle_step(g, pre, T, ids, L, H, A, ngram, C, K, draft_from):
    """The draws against the oracle's (equal, or within rounding of a boundary), then
    acceptance and append from the GPU's draws exactly, then the next draft."""
    ys = g["argmax"]
    o = oracle.verify_sample(pre["logits"], pre["u"], pre["draft"], pre["dlen"], T)
    diff = np.argwhere(ys != o["sampled"])
    # a flat distribution over 128k tokens has CDF steps of ~1e-5, so a few fp32
    # draws per step land next to the exact one; each must be a boundary case
    assert len(diff) <= max(2, ys.size // 50), diff
    l64 = _f64(pre["logits_t"]) if len(diff) else None
    for b, i in diff:
        assert _valid_draw(l64[b, i], T, float(pre["u"][b, i]), int(ys[b, i])), (b, i)
    B, K1 = ys.shape
    V = pre["logits"].shape[2]
    onehot = np.zeros((B, K1, V), np.float32)
    np.put_along_axis(onehot, ys[..., None].astype(np.int64), 1.0, axis=2)
    ids_o, L_o = pre["ids"].copy(), pre["L"].copy()
    e = oracle.verify_greedy(onehot, pre["draft"], pre["dlen"], ids=ids_o, seq_len=L_o, kv_keep=True)
    for k_g, k_o in (("acc", "accept_len"), ("nxt", "next_token"), ("kv", "kv_keep_len")):
        assert np.array_equal(g[k_g], e[k_o]), k_g
    assert np.array_equal(host(ids), ids_o) and np.array_equal(host(L), L_o)
    _compare(g, ids_o, L_o, H, A, None, 0, ngram, C, K, draft_from, status0=e["status"])


@pytest.mark.parametrize("T,V,B,mode,shared,temp", [
    (4096, 3000, 16, "both", True, 1.0), (8000, 300, 12, "hidden", False, 0.7),
    (2048, 20, 10, "attention", True, 1.3), (30000, 20000, 8, "both", False, 1.0)])
def test_sample_draft_equals_separate_calls(lib, T, V, B, mode, shared, temp):
    rng = np.random.default_rng(T + V)
    gen = torch.Generator(device=DEV).manual_seed(T + 5)
    K, C, ngram, d, R = 10, 64, (1, 3), 128, 12
    T_cap = T + 12 * (K + 1)
    ids = rng.integers(0, V, size=(B, T_cap)).astype(np.int32)
    lens = rng.integers(2, T + 1, size=B)
    lens[0] = T_cap - 1                       # full within two steps (CAPACITY)
    lens[1] = T_cap + 5                       # out of range throughout (SEQ_LEN)
    lens[3] = 1                               # x_t alone
    lens[4] = 0                               # empty
    H = torch.randn((B, T_cap, d), generator=gen, device=DEV).to(torch.bfloat16) if mode != "attention" else None
    A = torch.rand((B, R, T_cap), generator=gen, device=DEV).to(torch.bfloat16) if mode != "hidden" else None
    draft_from = "attention" if mode == "attention" else "hidden"
    ids_a, L_a = i32(ids), i32(lens)
    ids_b, L_b = ids_a.clone(), L_a.clone()
    ix_a = torch.empty(pk.pldp_index_size(B, V), dtype=torch.uint8, device=DEV)
    ix_b = torch.empty_like(ix_a)
    pk.pldp_index_build(ids_a, L_a, V, ix_a)
    pk.pldp_index_build(ids_b, L_b, V, ix_b)
    a, b_ = Buffers(B, K, V, C, DEV), Buffers(B, K, V, C, DEV)
    _draft(a, ids_a, L_a, ix_a, V, H, A, ngram, draft_from)
    _draft(b_, ids_b, L_b, ix_b, V, H, A, ngram, draft_from)
    st = np.zeros(B, np.uint32)
    accepted = 0
    for step in range(5):
        # logits that favour the draft (its tokens get +12) so that drafts are partly accepted
        logits = torch.randn((B, K + 1, V), generator=gen, device=DEV) * 1.5
        dr = b_.draft.clamp(0, V - 1).long()
        logits[:, :K].scatter_add_(2, dr[:, :, None], torch.full((B, K, 1), 12.0, device=DEV))
        logits = logits.to(torch.bfloat16)
        u = torch.rand((B, K + 1), generator=gen, device=DEV)
        if step == 2:
            a.dlen[2] = K + 3                 # an out-of-range draft length (DRAFT_LEN, clamped)
            b_.dlen[2] = K + 3
        pre = dict(ids=host(ids_b), L=host(L_b), logits=host(logits), logits_t=logits, u=host(u),
                   draft=host(b_.draft), dlen=host(b_.dlen))
        a.status.zero_()
        b_.status.zero_()
        _separate(a, logits, u, temp, ids_a, L_a, ix_a, V, H, A, ngram, draft_from)
        _fused(b_, logits, u, temp, ids_b, L_b, ix_b, V, H, A, ngram, draft_from, shared=shared)
        torch.cuda.synchronize()
        g = _snap(b_)
        _same(_snap(a), g, step)
        assert torch.equal(ids_a, ids_b) and torch.equal(L_a, L_b), step
        _same_index(ix_a, ix_b, B, V)
        _oracle_step(g, pre, temp, ids_b, L_b, H, A, ngram, C, K, draft_from)
        st |= g["status"].view(np.uint32)
        accepted += int(g["acc"].sum())
    assert st[0] & pk.PLDP_ST_CAPACITY and st[1] & pk.PLDP_ST_SEQ_LEN and st[2] & pk.PLDP_ST_DRAFT_LEN
    assert st[4] & pk.PLDP_ST_SEQ_LEN and host(L_b)[4] == 0
    assert accepted > 0                       # drafts were (partly) accepted


def test_sample_draft_decode_loop(lib):
    """A sustained loop (batch 32, context 4096, V 128256, both rankings) at T = 1:
    each step samples and drafts the next with the fused call on one copy of the
    state and with the two calls on another."""
    w = wl.CONFIGS["decode_loop_b128_ctx32k"].replace(B=32, prompt_len=3072, out_len=1024, d=512)
    steps = 6
    loop = wl.DecodeLoop(w, steps=steps, device=DEV)
    B, K, C, V = w.B, w.K, w.C_cap, w.V
    ng = (w.ngram_min, w.ngram_max)
    ids_b, L_b = loop.ids.clone(), loop.seq_len.clone()
    ix_a = torch.empty(pk.pldp_index_size(B, V), dtype=torch.uint8, device=DEV)
    ix_b = torch.empty_like(ix_a)
    pk.pldp_index_build(loop.ids, loop.seq_len, V, ix_a)
    pk.pldp_index_build(ids_b, L_b, V, ix_b)
    a, b_ = Buffers(B, K, V, C, DEV), Buffers(B, K, V, C, DEV)
    loop.step_inputs(0)
    _draft(a, loop.ids, loop.seq_len, ix_a, V, loop.H, loop.A, ng, "hidden")
    _draft(b_, ids_b, L_b, ix_b, V, loop.H, loop.A, ng, "hidden")
    gen = torch.Generator(device=DEV).manual_seed(9)
    for s in range(steps):
        loop.step_inputs(s)
        u = torch.rand((B, K + 1), generator=gen, device=DEV)
        pre = dict(ids=host(ids_b), L=host(L_b), logits=host(loop.logits), logits_t=loop.logits, u=host(u),
                   draft=host(b_.draft), dlen=host(b_.dlen))
        a.status.zero_()
        b_.status.zero_()
        _separate(a, loop.logits, u, 1.0, loop.ids, loop.seq_len, ix_a, V, loop.H, loop.A, ng, "hidden")
        _fused(b_, loop.logits, u, 1.0, ids_b, L_b, ix_b, V, loop.H, loop.A, ng, "hidden")
        torch.cuda.synchronize()
        g = _snap(b_)
        _same(_snap(a), g, s)
        assert torch.equal(loop.ids, ids_b) and torch.equal(loop.seq_len, L_b)
        _same_index(ix_a, ix_b, B, V)
        _oracle_step(g, pre, 1.0, ids_b, L_b, loop.H, loop.A, ng, C, K, "hidden")
    assert (host(L_b) > w.T).all()


def test_sample_draft_graph_capture_replays(lib):
    """One pldp_verify_sample_draft call captured in a CUDA graph and replayed step
    after step gives the eager call's results, the token index kept up to date by the
    replays (the uniforms and logits are rewritten in place before each replay)."""
    w = wl.CONFIGS["decode_loop_b128_ctx32k"].replace(B=16, prompt_len=3000, out_len=1000, V=32000, d=1024)
    ng = (w.ngram_min, w.ngram_max)
    B, K, C, V = w.B, w.K, w.C_cap, w.V
    loops = [wl.DecodeLoop(w, steps=6, device=DEV) for _ in range(2)]
    bufs = [Buffers(B, K, V, C, DEV) for _ in range(2)]
    idx = [torch.empty(pk.pldp_index_size(B, V), dtype=torch.uint8, device=DEV) for _ in range(2)]
    wss = [torch.empty(pk.pldp_verify_sample_draft_workspace_size(B, K, V), dtype=torch.uint8, device=DEV)
           for _ in range(2)]
    us = [torch.zeros((B, K + 1), dtype=torch.float32, device=DEV) for _ in range(2)]

    def call(i, stream=None):
        lp, buf = loops[i], bufs[i]
        pk.pldp_verify_sample_draft(lp.logits, us[i], buf.draft, buf.dlen, buf.acc, buf.nxt, wss[i], lp.ids,
                                    lp.seq_len, ng[0], ng[1], buf.cand, buf.cnt, buf.ml, buf.draft, buf.dlen, idx[i],
                                    temperature=1.0, sampled=buf.argmax, kv_keep_len=buf.kv, stream=stream,
                                    **_kw(buf, lp.H, lp.A, "hidden"))

    for i in range(2):
        lp, buf = loops[i], bufs[i]
        pk.pldp_index_build(lp.ids, lp.seq_len, V, idx[i])
        lp.step_inputs(0)
        _draft(buf, lp.ids, lp.seq_len, idx[i], V, lp.H, lp.A, ng, "hidden")
    # the stats pass's launch shape is looked up once, on an uncaptured call
    tmp = torch.zeros(B, dtype=torch.int32, device=DEV)
    pk.pldp_verify_sample(loops[0].logits, us[0], bufs[0].draft, bufs[0].dlen, tmp, tmp.clone(),
                          torch.empty(pk.pldp_verify_sample_workspace_size(B, K, V), dtype=torch.uint8, device=DEV))
    torch.cuda.synchronize()
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        call(1, stream=torch.cuda.current_stream())
    gen = torch.Generator(device=DEV).manual_seed(4)
    for s in range(6):
        u = torch.rand((B, K + 1), generator=gen, device=DEV)
        for i in range(2):
            loops[i].step_inputs(s)
            us[i].copy_(u)
        call(0)
        graph.replay()
        torch.cuda.synchronize()
        ga, gb = _snap(bufs[0]), _snap(bufs[1])
        for k in ("cnt", "ml", "best_h", "best_a", "draft", "dlen", "acc", "nxt", "argmax", "kv", "status"):
            assert np.array_equal(ga[k], gb[k]), (s, k)
        assert torch.equal(loops[0].ids, loops[1].ids) and torch.equal(loops[0].seq_len, loops[1].seq_len)
        assert torch.equal(idx[0][:4 * B], idx[1][:4 * B])
