"""GPU parity at the full sizes of the five workloads, in the launch configuration
the benchmark uses.  Every output of every sequence is compared with the oracle
at every step: the integer outputs bit-exactly, the scores and choices of both
rankings by the parity rules.  The hidden and attention tensors are too large to
copy to the host whole (37.8 GB of hidden rows in the decode loop), so the oracle
is handed host arrays that hold exactly the rows its rankings read, for the
oracle's own candidate lists (tests._parity.oracle_rows)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from tests._parity import Buffers, check_choice, check_scores, gpu_step, host, oracle_rows, snapshot

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.mark.parametrize("fused", [False, True], ids=["calls", "fused"])
@pytest.mark.parametrize("name", ["one_step_b1_ctx512", "hidden_b8_ctx4k", "hidden_b64_ctx16k",
                                  "attention_b32_ctx8k"])
def test_single_step_config(lib, name, fused):
    w = wl.CONFIGS[name]
    inp = wl.single_step(w, device=DEV)
    B, K, C = w.B, w.K, w.C_cap
    ids0, L0 = host(inp["ids"]), host(inp["seq_len"])
    buf = Buffers(B, K, w.V, C, DEV)
    draft_from = "hidden" if inp["H"] is not None else "attention"
    gpu_step(buf, inp["ids"], inp["seq_len"], inp["logits"], ngram=(w.ngram_min, w.ngram_max),
             H=inp["H"], A=inp["A"], row_idx=None, draft_from=draft_from, fused=fused)
    g = snapshot(buf)

    o_cand, o_cnt, o_ml, o_st = oracle.find_candidates(ids0, L0, w.ngram_min, w.ngram_max, C)
    assert np.array_equal(g["cnt"], o_cnt) and np.array_equal(g["ml"], o_ml)
    for b in range(B):
        n = min(o_cnt[b], C)
        assert np.array_equal(g["cand"][b, :n], o_cand[b, :n])
    Hs, As = oracle_rows(inp["H"], inp["A"], L0, o_cand, o_cnt)
    if inp["H"] is not None:
        o_s, o_b, _ = oracle.rank_hidden(Hs, L0, o_cand, o_cnt)
        check_scores(g["scores_h"], o_s, o_cnt, C)
        check_choice(g["best_h"], o_b, o_s, o_cand, o_cnt, C)
    if inp["A"] is not None:
        o_s, o_b, _ = oracle.rank_attention(As, L0, o_cand, o_cnt)
        check_scores(g["scores_a"], o_s, o_cnt, C)
        assert np.array_equal(g["best_a"], o_b)
    best = g["best_h"] if draft_from == "hidden" else g["best_a"]
    o_d, o_dl = oracle.extract_draft(ids0, L0, best, K)
    assert np.array_equal(g["draft"], o_d) and np.array_equal(g["dlen"], o_dl)
    ids_o, L_o = ids0.copy(), L0.copy()
    o = oracle.verify_greedy(host(inp["logits"]), o_d, o_dl, ids=ids_o, seq_len=L_o, kv_keep=True)
    for k_g, k_o in (("argmax", "argmax"), ("acc", "accept_len"), ("nxt", "next_token"),
                     ("kv", "kv_keep_len")):
        assert np.array_equal(g[k_g], o[k_o]), k_g
    assert np.array_equal(host(inp["ids"]), ids_o) and np.array_equal(host(inp["seq_len"]), L_o)
    assert (g["status"] == 0).all()
    # the planted structure is recovered: the planted accept length on (nearly) every sequence
    hit = float(np.mean(g["acc"] == inp["planted_accept"]))
    assert hit >= 0.8, hit
    if name == "one_step_b1_ctx512":
        assert g["acc"].tolist() == [6]


@pytest.mark.parametrize("fused", [False, True], ids=["calls", "fused"])
def test_decode_loop_full(lib, fused):
    """The sustained loop: every step compared with the oracle run on the same
    pre-step state; the emitted streams equal the ground truth (losslessness)."""
    w = wl.CONFIGS["decode_loop_b128_ctx32k"]
    steps = 5
    loop = wl.DecodeLoop(w, steps=steps, device=DEV)
    B, K, C = w.B, w.K, w.C_cap
    buf = Buffers(B, K, w.V, C, DEV)
    for s in range(steps):
        loop.step_inputs(s)
        ids0, L0 = host(loop.ids), host(loop.seq_len)
        lg = host(loop.logits)
        o_cand, o_cnt, o_ml, _ = oracle.find_candidates(ids0, L0, w.ngram_min, w.ngram_max, C)
        Hs, As = oracle_rows(loop.H, loop.A, L0, o_cand, o_cnt)
        gpu_step(buf, loop.ids, loop.seq_len, loop.logits, ngram=(w.ngram_min, w.ngram_max), H=loop.H,
                 A=loop.A, draft_from="hidden", fused=fused)
        g = snapshot(buf)
        assert np.array_equal(g["cnt"], o_cnt) and np.array_equal(g["ml"], o_ml)
        for b in range(B):
            n = min(o_cnt[b], C)
            assert np.array_equal(g["cand"][b, :n], o_cand[b, :n])
        o_s, o_b, _ = oracle.rank_hidden(Hs, L0, o_cand, o_cnt)
        check_scores(g["scores_h"], o_s, o_cnt, C)
        check_choice(g["best_h"], o_b, o_s, o_cand, o_cnt, C)
        o_sa, o_ba, _ = oracle.rank_attention(As, L0, o_cand, o_cnt)
        check_scores(g["scores_a"], o_sa, o_cnt, C)
        assert np.array_equal(g["best_a"], o_ba)
        o_d, o_dl = oracle.extract_draft(ids0, L0, g["best_h"], K)
        assert np.array_equal(g["draft"], o_d) and np.array_equal(g["dlen"], o_dl)
        ids_o, L_o = ids0.copy(), L0.copy()
        o = oracle.verify_greedy(lg, o_d, o_dl, ids=ids_o, seq_len=L_o, kv_keep=True)
        assert np.array_equal(g["argmax"], o["argmax"]) and np.array_equal(g["acc"], o["accept_len"])
        assert np.array_equal(g["nxt"], o["next_token"]) and np.array_equal(g["kv"], o["kv_keep_len"])
        assert np.array_equal(host(loop.ids), ids_o) and np.array_equal(host(loop.seq_len), L_o)
        assert (g["status"] == 0).all()
    L = host(loop.seq_len)
    ids, gt = host(loop.ids), loop.gt_host
    for b in range(B):
        assert np.array_equal(ids[b, :L[b]], gt[b, :L[b]]), b
    assert (L - w.T).mean() > steps * 1.5      # drafts are accepted: more than one token per step


@pytest.mark.parametrize("fused", [False, True], ids=["calls", "fused"])
def test_graph_capture_replays_the_step(lib, fused):
    """The five calls captured in one CUDA graph give the eager results, and the
    verify workspace returns to zero between replays."""
    w = wl.CONFIGS["decode_loop_b128_ctx32k"].replace(B=16, prompt_len=3000, out_len=1000, V=32000, d=1024)
    a = wl.DecodeLoop(w, steps=6, device=DEV)
    b = wl.DecodeLoop(w, steps=6, device=DEV)
    buf_a = Buffers(w.B, w.K, w.V, w.C_cap, DEV)
    buf_b = Buffers(w.B, w.K, w.V, w.C_cap, DEV)
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    b.step_inputs(0)
    torch.cuda.synchronize()
    with torch.cuda.graph(graph, stream=stream):
        gpu_step(buf_b, b.ids, b.seq_len, b.logits, H=b.H, A=b.A, stream=torch.cuda.current_stream(),
                 fused=fused)
    b.reset()
    for s in range(6):
        a.step_inputs(s)
        b.step_inputs(s)
        gpu_step(buf_a, a.ids, a.seq_len, a.logits, H=a.H, A=a.A, fused=fused)
        graph.replay()
        torch.cuda.synchronize()
        ga, gb = snapshot(buf_a), snapshot(buf_b)
        for k in ("cnt", "best_h", "best_a", "draft", "acc", "nxt", "argmax"):
            assert np.array_equal(ga[k], gb[k]), (s, k)
        assert torch.equal(a.ids, b.ids) and torch.equal(a.seq_len, b.seq_len)
        assert int(buf_b.ws.count_nonzero()) == 0


def test_graph_capture_replays_verify_draft(lib):
    """One pldp_verify_greedy_draft call captured in a CUDA graph and replayed step after
    step gives the eager call's results, with the token index kept up to date by the
    replays; the verify workspace returns to zero between replays."""
    import paper_2412_01447_gb300 as pk
    w = wl.CONFIGS["decode_loop_b128_ctx32k"].replace(B=16, prompt_len=3000, out_len=1000, V=32000, d=1024)
    ng = (w.ngram_min, w.ngram_max)
    loops = [wl.DecodeLoop(w, steps=6, device=DEV) for _ in range(2)]
    bufs = [Buffers(w.B, w.K, w.V, w.C_cap, DEV) for _ in range(2)]
    idx = [torch.empty(pk.pldp_index_size(w.B, w.V), dtype=torch.uint8, device=DEV) for _ in range(2)]

    def kw(lp, buf):
        return dict(H=lp.H, best_h=buf.best_h, A=lp.A, best_a=buf.best_a, draft_from="hidden", status=buf.status)

    def call(i, stream=None):
        lp, buf = loops[i], bufs[i]
        pk.pldp_verify_greedy_draft(lp.logits, buf.draft, buf.dlen, buf.acc, buf.nxt, buf.ws, lp.ids, lp.seq_len,
                                    ng[0], ng[1], buf.cand, buf.cnt, buf.ml, buf.draft, buf.dlen, idx[i],
                                    argmax=buf.argmax, kv_keep_len=buf.kv, stream=stream, **kw(lp, buf))

    for i in range(2):                        # the index and the first draft of each copy
        lp, buf = loops[i], bufs[i]
        pk.pldp_index_build(lp.ids, lp.seq_len, w.V, idx[i])
        lp.step_inputs(0)
        pk.pldp_draft_step(lp.ids, lp.seq_len, ng[0], ng[1], buf.cand, buf.cnt, buf.ml, w.K, buf.draft, buf.dlen,
                           None, index=idx[i], V=w.V, **kw(lp, buf))
    torch.cuda.synchronize()
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        call(1, stream=torch.cuda.current_stream())
    for s in range(6):
        for i in range(2):
            loops[i].step_inputs_next(s, bufs[i].draft, bufs[i].dlen)
        call(0)
        graph.replay()
        torch.cuda.synchronize()
        ga, gb = snapshot(bufs[0]), snapshot(bufs[1])
        for k in ("cnt", "ml", "best_h", "best_a", "draft", "dlen", "acc", "nxt", "argmax", "kv", "status"):
            assert np.array_equal(ga[k], gb[k]), (s, k)
        assert torch.equal(loops[0].ids, loops[1].ids) and torch.equal(loops[0].seq_len, loops[1].seq_len)
        assert torch.equal(idx[0][:4 * w.B], idx[1][:4 * w.B])
        assert int(bufs[1].ws.count_nonzero()) == 0


def test_decode_loop_full_verify_draft(lib):
    """The benchmark's configuration: the full decode loop (batch 128, context 32768)
    with one pldp_verify_greedy_draft call per step (verification, then the next draft
    with the token index).  Each step is compared with the oracle: verification of the
    GPU's draft on the pre-step state, then candidates, rankings and draft of every
    sequence on the state it leaves."""
    import paper_2412_01447_gb300 as pk
    w = wl.CONFIGS["decode_loop_b128_ctx32k"]
    steps = 4
    loop = wl.DecodeLoop(w, steps=steps, device=DEV)
    B, K, C = w.B, w.K, w.C_cap
    ng = (w.ngram_min, w.ngram_max)
    buf = Buffers(B, K, w.V, C, DEV)
    index = torch.empty(pk.pldp_index_size(B, w.V), dtype=torch.uint8, device=DEV)
    pk.pldp_index_build(loop.ids, loop.seq_len, w.V, index)
    kw = dict(H=loop.H, best_h=buf.best_h, h_scores=buf.scores_h, best_h_score=buf.bscore_h, A=loop.A,
              best_a=buf.best_a, a_scores=buf.scores_a, best_a_score=buf.bscore_a, draft_from="hidden",
              status=buf.status)

    def oracle_draft_inputs(ids0, L0):
        """The oracle's candidates on this state, and the rows its rankings read."""
        o = oracle.find_candidates(ids0, L0, ng[0], ng[1], C)
        return o, oracle_rows(loop.H, loop.A, L0, o[0], o[1])

    def check_draft(ids0, L0, o_fc, rows):
        g = snapshot(buf)
        o_cand, o_cnt, o_ml, _ = o_fc
        Hs, As = rows
        assert np.array_equal(g["cnt"], o_cnt) and np.array_equal(g["ml"], o_ml)
        for b in range(B):
            n = min(o_cnt[b], C)
            assert np.array_equal(g["cand"][b, :n], o_cand[b, :n]), b
        o_s, o_b, _ = oracle.rank_hidden(Hs, L0, o_cand, o_cnt)
        check_scores(g["scores_h"], o_s, o_cnt, C)
        check_choice(g["best_h"], o_b, o_s, o_cand, o_cnt, C)
        o_sa, o_ba, _ = oracle.rank_attention(As, L0, o_cand, o_cnt)
        check_scores(g["scores_a"], o_sa, o_cnt, C)
        assert np.array_equal(g["best_a"], o_ba)
        o_d, o_dl = oracle.extract_draft(ids0, L0, g["best_h"], K)
        assert np.array_equal(g["draft"], o_d) and np.array_equal(g["dlen"], o_dl)
        return g

    loop.step_inputs(0)                       # the first draft, as a prefill would make it
    ids0, L0 = host(loop.ids), host(loop.seq_len)
    o_fc, rows = oracle_draft_inputs(ids0, L0)
    pk.pldp_draft_step(loop.ids, loop.seq_len, ng[0], ng[1], buf.cand, buf.cnt, buf.ml, K, buf.draft, buf.dlen,
                       None, index=index, V=w.V, **kw)
    check_draft(ids0, L0, o_fc, rows)
    for s in range(steps):
        loop.step_inputs_next(s, buf.draft, buf.dlen)
        ids0, L0, lg = host(loop.ids), host(loop.seq_len), host(loop.logits)
        d0, dl0 = host(buf.draft), host(buf.dlen)
        ids_o, L_o = ids0.copy(), L0.copy()
        o = oracle.verify_greedy(lg, d0, dl0, ids=ids_o, seq_len=L_o, kv_keep=True)
        o_fc, rows = oracle_draft_inputs(ids_o, L_o)   # the oracle's next draft inputs, on the state it left
        pk.pldp_verify_greedy_draft(loop.logits, buf.draft, buf.dlen, buf.acc, buf.nxt, buf.ws, loop.ids,
                                    loop.seq_len, ng[0], ng[1], buf.cand, buf.cnt, buf.ml, buf.draft, buf.dlen,
                                    index, argmax=buf.argmax, kv_keep_len=buf.kv, **kw)
        g = check_draft(ids_o, L_o, o_fc, rows)       # the next draft, on the state verification left
        assert np.array_equal(g["argmax"], o["argmax"]) and np.array_equal(g["acc"], o["accept_len"])
        assert np.array_equal(g["nxt"], o["next_token"]) and np.array_equal(g["kv"], o["kv_keep_len"])
        assert np.array_equal(host(loop.ids), ids_o) and np.array_equal(host(loop.seq_len), L_o)
        assert (g["status"] == 0).all()
    L = host(loop.seq_len)
    ids, gt = host(loop.ids), loop.gt_host
    for b in range(B):
        assert np.array_equal(ids[b, :L[b]], gt[b, :L[b]]), b
    assert (L - w.T).mean() > steps * 1.5
