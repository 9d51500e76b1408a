"""pldp_verify_greedy_draft (verification of a step, then the next step's drafting
with the token index, in one call) against pldp_verify_greedy followed by
pldp_draft_step on the same state: every output, the extended contexts and the
index must agree bit for bit, step after step, and every output equals the
oracle's (verification on the pre-step state, then the next draft on the state
it leaves).  Covers random contexts (few and
many occurrences, the rescan fallback), a context that runs out of capacity, an
out-of-range length, an out-of-range draft length, the draft buffers shared
between the two halves or not, and a sustained decode loop."""
import numpy as np
import pytest
import torch

import oracle
import paper_2412_01447_gb300 as pk
import workloads as wl
from tests._parity import Buffers, host, snapshot
from tests.test_gpu_fused import _compare

pytestmark = pytest.mark.gpu
DEV = "cuda"
OUT = ("cand", "cnt", "ml", "status", "best_h", "best_a", "scores_h", "scores_a", "bscore_h", "bscore_a",
       "draft", "dlen", "acc", "nxt", "kv", "argmax")


def i32(x):
    return torch.as_tensor(np.asarray(x, np.int32), device=DEV)


def _kw(buf, H, A, draft_from):
    return dict(H=H, best_h=buf.best_h if H is not None else None, h_scores=buf.scores_h,
                best_h_score=buf.bscore_h, A=A, best_a=buf.best_a if A is not None else None,
                a_scores=buf.scores_a, best_a_score=buf.bscore_a, draft_from=draft_from, status=buf.status)


def _draft(buf, ids, L, index, V, H, A, ngram, draft_from):
    pk.pldp_draft_step(ids, L, ngram[0], ngram[1], buf.cand, buf.cnt, buf.ml, buf.draft.shape[1], buf.draft,
                       buf.dlen, None, index=index, V=V, **_kw(buf, H, A, draft_from))


def _separate(buf, logits, ids, L, index, V, H, A, ngram, draft_from):
    pk.pldp_verify_greedy(logits, buf.draft, buf.dlen, buf.acc, buf.nxt, buf.ws, argmax=buf.argmax, ids=ids,
                          seq_len=L, kv_keep_len=buf.kv, status=buf.status)
    _draft(buf, ids, L, index, V, H, A, ngram, draft_from)


def _fused(buf, logits, ids, L, index, V, H, A, ngram, draft_from, shared=True):
    if shared:
        nd, nl = buf.draft, buf.dlen
    else:
        nd, nl = torch.full_like(buf.draft, -7), torch.full_like(buf.dlen, -7)
    pk.pldp_verify_greedy_draft(logits, buf.draft, buf.dlen, buf.acc, buf.nxt, buf.ws, ids, L, ngram[0], ngram[1],
                                buf.cand, buf.cnt, buf.ml, nd, nl, index, argmax=buf.argmax, kv_keep_len=buf.kv,
                                **_kw(buf, H, A, draft_from))
    if not shared:
        buf.draft.copy_(nd)
        buf.dlen.copy_(nl)


def _snap(buf):
    s = snapshot(buf)
    for k in ("acc", "nxt", "kv", "argmax"):
        s[k] = host(getattr(buf, k))
    return s


def _same(a, b, what):
    for k in OUT:
        assert np.array_equal(a[k], b[k], equal_nan=True), (what, k)


def _same_index(x, y, B, V):
    """Two token indexes hold the same thing: the indexed lengths, per entry the count,
    and the set of positions of every entry that holds them all (count <= 15).  Which
    slot a position takes, and which positions an overfull entry keeps, depend on the
    order in which equal tokens inserted together took their atomics; lookups do not."""
    up = lambda n: (n + 255) // 256 * 256
    off = 2 * up(4 * B)
    assert torch.equal(x[:4 * B], y[:4 * B])
    ex = x[off:off + B * V * 64].view(torch.int32).view(B, V, 16)
    ey = y[off:off + B * V * 64].view(torch.int32).view(B, V, 16)
    assert torch.equal(ex[..., 0], ey[..., 0])
    k = torch.arange(15, device=x.device)
    keep = (k[None, None] < ex[..., :1]) & (ex[..., :1] <= 15)
    sx = torch.where(keep, ex[..., 1:], torch.full_like(ex[..., 1:], 1 << 30)).sort(dim=-1).values
    sy = torch.where(keep, ey[..., 1:], torch.full_like(ey[..., 1:], 1 << 30)).sort(dim=-1).values
    assert torch.equal(sx, sy)


def _oracle_step(g, pre, ids, L, H, A, ngram, C, K, draft_from):
    """The fused call's outputs g against the oracle: greedy verification of the
    pre-step draft on the pre-step state, then the next draft on the state that
    verification leaves (every status bit of both halves)."""
    ids_o, L_o = pre["ids"].copy(), pre["L"].copy()
    o = oracle.verify_greedy(pre["logits"], pre["draft"], pre["dlen"], ids=ids_o, seq_len=L_o, kv_keep=True)
    for k_g, k_o in (("argmax", "argmax"), ("acc", "accept_len"), ("nxt", "next_token"), ("kv", "kv_keep_len")):
        assert np.array_equal(g[k_g], o[k_o]), k_g
    assert np.array_equal(host(ids), ids_o) and np.array_equal(host(L), L_o)
    _compare(g, ids_o, L_o, H, A, None, 0, ngram, C, K, draft_from, status0=o["status"])


def _planted_logits(draft, dlen, V, gen, accept):
    """bf16 logits [B, K+1, V]: N(0,1), with row i's maximum moved onto draft[b, i] for
    i < accept[b] (the step accepts min(accept, draft_len) tokens, fewer where a draft
    token is out of range)."""
    B, K = draft.shape
    lg = torch.randn((B, K + 1, V), generator=gen, device=DEV)
    i = torch.arange(K, device=DEV)[None]
    ok = (i < accept[:, None]) & (i < dlen[:, None]) & (draft >= 0) & (draft < V)
    top = lg[:, :K].amax(dim=2) + 1.0
    rows = lg[:, :K]
    rows.scatter_(2, draft.clamp(0, V - 1).long()[:, :, None],
                  torch.where(ok, top, rows.gather(2, draft.clamp(0, V - 1).long()[:, :, None])[:, :, 0])[:, :, None])
    return lg.to(torch.bfloat16)


@pytest.mark.parametrize("T,V,B,mode,shared", [
    (4096, 3000, 16, "both", True), (8000, 300, 12, "hidden", False), (2048, 20, 10, "attention", True),
    (30000, 20000, 8, "both", False)])
def test_verify_draft_equals_separate_calls(lib, T, V, B, mode, shared):
    _verify_draft_case(T, V, B, mode, shared, K=10, C=64, ngram=(1, 3), dt=torch.bfloat16)


@pytest.mark.parametrize("K,C,ngram,dt", [(40, 64, (1, 3), torch.bfloat16), (6, 2, (2, 4), torch.float32),
                                          (33, 8, (1, 8), torch.float32)])
def test_verify_draft_other_shapes(lib, K, C, ngram, dt):
    """Drafts longer than the staged window (K > 32), short candidate lists, other
    n-gram ranges, and fp32 hidden rows and attention values."""
    _verify_draft_case(6000, 2000, 12, "both", True, K=K, C=C, ngram=ngram, dt=dt)


def _verify_draft_case(T, V, B, mode, shared, K, C, ngram, dt):
    rng = np.random.default_rng(T + V + K)
    gen = torch.Generator(device=DEV).manual_seed(T + 3)
    d, R = 128, 12
    T_cap = T + 12 * (K + 1)
    ids = rng.integers(0, V, size=(B, T_cap)).astype(np.int32)
    lens = rng.integers(2, T + 1, size=B)
    lens[0] = T_cap - 1                       # full within two steps (CAPACITY)
    lens[1] = T_cap + 5                       # out of range throughout (SEQ_LEN)
    lens[3] = 1                               # x_t alone: no H_{t-1}, nothing before it
    lens[4] = 0                               # empty: verification refuses it (SEQ_LEN), drafting finds nothing
    H = torch.randn((B, T_cap, d), generator=gen, device=DEV).to(dt) if mode != "attention" else None
    A = torch.rand((B, R, T_cap), generator=gen, device=DEV).to(dt) if mode != "hidden" else None
    if A is not None and T % 3 == 0:                  # key-major: the R values of a key side by side
        A = A.transpose(1, 2).contiguous().transpose(1, 2)
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
    for step in range(6):
        accept = torch.as_tensor(rng.integers(0, K + 1, size=B), device=DEV)
        if step == 2:
            a.dlen[2] = K + 3                 # an out-of-range draft length (DRAFT_LEN, clamped)
            b_.dlen[2] = K + 3
        logits = _planted_logits(a.draft, a.dlen, V, gen, accept)
        pre = dict(ids=host(ids_b), L=host(L_b), logits=host(logits), draft=host(b_.draft), dlen=host(b_.dlen))
        a.status.zero_()
        b_.status.zero_()
        _separate(a, logits, ids_a, L_a, ix_a, V, H, A, ngram, draft_from)
        _fused(b_, logits, ids_b, L_b, ix_b, V, H, A, ngram, draft_from, shared=shared)
        torch.cuda.synchronize()
        g = _snap(b_)
        _same(_snap(a), g, step)
        assert torch.equal(ids_a, ids_b) and torch.equal(L_a, L_b), step
        _same_index(ix_a, ix_b, B, V)
        _oracle_step(g, pre, ids_b, L_b, H, A, ngram, C, K, draft_from)
        st |= g["status"].view(np.uint32)
    assert st[0] & pk.PLDP_ST_CAPACITY and st[1] & pk.PLDP_ST_SEQ_LEN and st[2] & pk.PLDP_ST_DRAFT_LEN
    assert st[4] & pk.PLDP_ST_SEQ_LEN and host(L_b)[4] == 0 and host(L_b)[3] > 1
    for ix in (ix_a, ix_b):                   # the empty context's index stays usable (nothing indexed)
        assert host(ix[:4 * B].view(torch.int32))[4] == 0
    assert (host(b_.ws) == 0).all()           # the verification workspace is left zero


def test_verify_draft_decode_loop(lib):
    """The sustained loop (batch 32, context 4096, V 128256): each step verifies and
    drafts the next with the fused call on one copy of the state and with the two
    calls on another; the emitted streams are the ground truth."""
    w = wl.CONFIGS["decode_loop_b128_ctx32k"].replace(B=32, prompt_len=3072, out_len=1024, d=512)
    steps = 6
    loop = wl.DecodeLoop(w, steps=steps, device=DEV)
    B, K, C = w.B, w.K, w.C_cap
    ids_b, L_b = loop.ids.clone(), loop.seq_len.clone()
    ix_a = torch.empty(pk.pldp_index_size(B, w.V), dtype=torch.uint8, device=DEV)
    ix_b = torch.empty_like(ix_a)
    pk.pldp_index_build(loop.ids, loop.seq_len, w.V, ix_a)
    pk.pldp_index_build(ids_b, L_b, w.V, ix_b)
    a, b_ = Buffers(B, K, w.V, C, DEV), Buffers(B, K, w.V, C, DEV)
    loop.step_inputs(0)
    _draft(a, loop.ids, loop.seq_len, ix_a, w.V, loop.H, loop.A, (w.ngram_min, w.ngram_max), "hidden")
    _draft(b_, ids_b, L_b, ix_b, w.V, loop.H, loop.A, (w.ngram_min, w.ngram_max), "hidden")
    ng = (w.ngram_min, w.ngram_max)
    for s in range(steps):
        loop.step_inputs(s)                   # logits for this step (and attention rows, shared by both)
        pre = dict(ids=host(ids_b), L=host(L_b), logits=host(loop.logits), draft=host(b_.draft),
                   dlen=host(b_.dlen))
        a.status.zero_()
        b_.status.zero_()
        _separate(a, loop.logits, loop.ids, loop.seq_len, ix_a, w.V, loop.H, loop.A, ng, "hidden")
        _fused(b_, loop.logits, ids_b, L_b, ix_b, w.V, loop.H, loop.A, ng, "hidden")
        torch.cuda.synchronize()
        g = _snap(b_)
        _same(_snap(a), g, s)
        assert torch.equal(loop.ids, ids_b) and torch.equal(loop.seq_len, L_b)
        _same_index(ix_a, ix_b, B, w.V)
        _oracle_step(g, pre, ids_b, L_b, loop.H, loop.A, ng, C, K, "hidden")
    L = host(L_b)
    ids, gt = host(ids_b), loop.gt_host
    for b in range(B):
        assert np.array_equal(ids[b, :L[b]], gt[b, :L[b]]), b
