"""Helpers for the GPU parity tests: run one PLD+ step through the C ABI and the
same step through the oracle, and compare by the parity rules:

* candidate lists, counts, n-gram lengths, drafts, argmaxes, accept lengths,
  next tokens and appended contexts: bit-exact;
* scores: within SCORE_TOL absolute of the fp64 oracle;
* the chosen candidate: the oracle's own, or one whose oracle score is within
  SCORE_TOL of the oracle's best (a near tie that fp32 may order differently);
  the draft is then compared with the oracle's draft FOR THE GPU'S CHOICE and
  verification with the oracle's verification OF THE GPU'S DRAFT.
"""
import numpy as np
import torch

import oracle
import paper_2412_01447_gb300 as pk

SCORE_TOL = 2e-3


def host(t):
    """Exact host copy: bf16 -> uint16 bit patterns, others as numpy."""
    if t is None:
        return None
    if t.dtype == torch.bfloat16:
        return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    return t.contiguous().cpu().numpy()


class Buffers:
    def __init__(self, B, K, V, C_cap, device):
        i32 = dict(dtype=torch.int32, device=device)
        self.cand = torch.full((B, C_cap), -1, **i32)
        self.cnt = torch.zeros(B, **i32)
        self.ml = torch.zeros(B, **i32)
        self.status = torch.zeros(B, **i32)
        self.best_h = torch.zeros(B, **i32)
        self.best_a = torch.zeros(B, **i32)
        self.scores_h = torch.full((B, C_cap), float("nan"), dtype=torch.float32, device=device)
        self.scores_a = torch.full((B, C_cap), float("nan"), dtype=torch.float32, device=device)
        self.bscore_h = torch.zeros(B, dtype=torch.float32, device=device)
        self.bscore_a = torch.zeros(B, dtype=torch.float32, device=device)
        self.draft = torch.zeros((B, K), **i32)
        self.dlen = torch.zeros(B, **i32)
        self.argmax = torch.zeros((B, K + 1), **i32)
        self.acc = torch.zeros(B, **i32)
        self.nxt = torch.zeros(B, **i32)
        self.kv = torch.zeros(B, **i32)
        self.ws = torch.zeros(pk.pldp_verify_workspace_size(B, K, V), dtype=torch.uint8, device=device)
        self.dws = torch.zeros(pk.pldp_draft_workspace_size(B), dtype=torch.uint8, device=device)


def gpu_step(buf, ids, seq_len, logits, ngram=(1, 3), H=None, A=None, row_idx=None,
             agg=pk.PLDP_AGG_MAX, draft_from="hidden", threshold=float("-inf"), append=True,
             stream=None, fused=False):
    """One step through the C ABI; ids/seq_len are updated in place when append.
    fused: the drafting half runs as the single pldp_draft_step launch."""
    if fused:
        ri = None if row_idx is None or A is None else torch.as_tensor(row_idx, dtype=torch.int32,
                                                                        device=A.device)
        pk.pldp_draft_step(ids, seq_len, ngram[0], ngram[1], buf.cand, buf.cnt, buf.ml, buf.draft.shape[1],
                           buf.draft, buf.dlen, buf.dws, H=H, best_h=buf.best_h if H is not None else None,
                           h_scores=buf.scores_h, best_h_score=buf.bscore_h, threshold=threshold, A=A,
                           best_a=buf.best_a if A is not None else None, row_idx=ri, agg=agg,
                           a_scores=buf.scores_a, best_a_score=buf.bscore_a, draft_from=draft_from,
                           status=buf.status, stream=stream)
        if logits is not None:
            pk.pldp_verify_greedy(logits, buf.draft, buf.dlen, buf.acc, buf.nxt, buf.ws,
                                  argmax=buf.argmax, ids=ids if append else None,
                                  seq_len=seq_len if append else None,
                                  kv_keep_len=buf.kv if append else None, status=buf.status,
                                  stream=stream)
        return
    pk.pldp_find_candidates(ids, seq_len, ngram[0], ngram[1], buf.cand, buf.cnt, buf.ml,
                            buf.status, stream=stream)
    if H is not None:
        pk.pldp_rank_hidden(H, seq_len, buf.cand, buf.cnt, buf.best_h, scores=buf.scores_h,
                            best_score=buf.bscore_h, threshold=threshold, status=buf.status,
                            stream=stream)
    if A is not None:
        ri = None if row_idx is None else torch.as_tensor(row_idx, dtype=torch.int32,
                                                           device=A.device)
        pk.pldp_rank_attention(A, seq_len, buf.cand, buf.cnt, buf.best_a, row_idx=ri, agg=agg,
                               scores=buf.scores_a, best_score=buf.bscore_a, status=buf.status,
                               stream=stream)
    best = buf.best_h if draft_from == "hidden" else buf.best_a
    pk.pldp_extract_draft(ids, seq_len, best, buf.draft, buf.dlen, stream=stream)
    if logits is not None:
        pk.pldp_verify_greedy(logits, buf.draft, buf.dlen, buf.acc, buf.nxt, buf.ws, argmax=buf.argmax,
                              ids=ids if append else None, seq_len=seq_len if append else None,
                              kv_keep_len=buf.kv if append else None, status=buf.status,
                              stream=stream)


def oracle_rows(H, A, seq_len, cand, cnt):
    """Host copies of H [B, T_cap, d] and A [B, R, T_cap] (device tensors, or None)
    that hold exactly what the oracle's rankings read for these candidate lists: per
    sequence the query row H_{t-1} and each listed candidate's H_{j-1}, and each
    listed candidate's key column A[:, j].  The rest of each host array is zero
    pages that are never touched, so full-size tensors fit in host memory.  The
    candidate lists are the oracle's own (never the GPU's)."""
    B = len(seq_len)
    bh, rh, ba, ja = [], [], [], []
    for b in range(B):
        L = int(seq_len[b])
        T_cap = (H if H is not None else A).shape[1 if H is not None else 2]
        t = L - 1
        if t < 1 or L > T_cap:
            continue
        n = max(0, min(int(cnt[b]), cand.shape[1]))
        js = cand[b, :n].astype(np.int64)
        js = js[(js >= 0) & (js < t)]
        rows = np.unique(np.concatenate([js[js >= 1] - 1, [t - 1]]))
        bh += [b] * rows.size
        rh += rows.tolist()
        ba += [b] * js.size
        ja += js.tolist()
    Hs = As = None
    if H is not None:
        Hs = np.zeros(tuple(H.shape), np.uint16 if H.dtype == torch.bfloat16 else np.float32)
        if bh:
            bi, ri = np.asarray(bh), np.asarray(rh)
            Hs[bi, ri] = host(H[torch.as_tensor(bi, device=H.device), torch.as_tensor(ri, device=H.device)])
    if A is not None:
        As = np.zeros(tuple(A.shape), np.uint16 if A.dtype == torch.bfloat16 else np.float32)
        if ba:
            bi, ji = np.asarray(ba), np.asarray(ja)
            As[bi, :, ji] = host(A[torch.as_tensor(bi, device=A.device), :, torch.as_tensor(ji, device=A.device)])
    return Hs, As


def snapshot(buf):
    torch.cuda.synchronize()
    return {k: host(v) for k, v in vars(buf).items() if k not in ("ws", "dws")}


def check_scores(g_scores, o_scores, cnt, C_cap, rows=None):
    rows = range(len(cnt)) if rows is None else rows
    for b in rows:
        n = max(0, min(int(cnt[b]), C_cap))
        g, o = g_scores[b, :n].astype(np.float64), o_scores[b, :n]
        inf = np.isinf(o)
        assert np.array_equal(np.isinf(g), inf), (b, g, o)
        assert np.array_equal(g[inf], o[inf])
        if (~inf).any():
            err = np.abs(g[~inf] - o[~inf]).max()
            assert err <= SCORE_TOL, (b, err)


def check_choice(g_best, o_best, o_scores, cand, cnt, C_cap, rows=None):
    """GPU choice = oracle choice, or within SCORE_TOL of it by the oracle's scores."""
    rows = range(len(g_best)) if rows is None else rows
    near = 0
    for b in rows:
        if g_best[b] == o_best[b]:
            continue
        assert g_best[b] >= 0 and o_best[b] >= 0, (b, g_best[b], o_best[b])
        n = max(0, min(int(cnt[b]), C_cap))
        lst = list(cand[b, :n])
        s_g = o_scores[b, lst.index(g_best[b])]
        s_o = o_scores[b, lst.index(o_best[b])]
        assert abs(s_g - s_o) <= SCORE_TOL, (b, s_g, s_o)
        near += 1
    return near
