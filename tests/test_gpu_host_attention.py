"""Attention rows kept in pinned host memory: the rankings read them in place
(only the selected rows' values at the candidate keys cross the link) and give
exactly the results of the same rows on the device, for the separate Eq. 2
ranking and for the one-launch drafting with the token index, in both memory
orders (each row's keys side by side, or the R values of each key)."""
import numpy as np
import pytest
import torch

import paper_2412_01447_gb300 as pk
from tests._parity import Buffers, snapshot

pytestmark = pytest.mark.gpu
DEV = "cuda"


# all rows of a key-major layout take the dense whole-vector form of Eq. 2 (MAX)
@pytest.mark.parametrize("layout,select", [("head", True), ("key", True), ("key", False)])
def test_rank_attention_reads_host_rows_in_place(lib, layout, select):
    rng = np.random.default_rng(4)
    B, R, T, C = 12, 32, 3000, 64
    A = torch.rand((B, R, T), device=DEV).to(torch.bfloat16)
    if layout == "key":
        A = A.transpose(1, 2).contiguous().transpose(1, 2)
    A_host = torch.empty_strided(A.shape, A.stride(), dtype=A.dtype, pin_memory=True)
    A_host.copy_(A)
    lens = torch.as_tensor(rng.integers(2, T + 1, size=B).astype(np.int32), device=DEV)
    cands = torch.as_tensor(np.sort(rng.choice(T - 1, (B, C)), axis=1).astype(np.int32), device=DEV)
    cnt = torch.as_tensor(rng.integers(0, C + 1, size=B).astype(np.int32), device=DEV)
    rows = torch.as_tensor(np.array([3, 7, 1, 30, 12], np.int32), device=DEV) if select else None
    out = []
    for src in (A, A_host):
        buf = Buffers(B, 4, 8, C, DEV)
        lib.pldp_rank_attention(src, lens, cands, cnt, buf.best_a, row_idx=rows, scores=buf.scores_a,
                                best_score=buf.bscore_a, status=buf.status)
        out.append(snapshot(buf))
    for k in ("best_a", "scores_a", "bscore_a", "status"):
        assert np.array_equal(out[0][k], out[1][k], equal_nan=True), k


def test_draft_step_reads_host_rows_in_place(lib):
    rng = np.random.default_rng(5)
    B, R, T, V, d, K = 16, 24, 5000, 300, 128, 8
    ids = torch.as_tensor(rng.integers(0, V, size=(B, T)).astype(np.int32), device=DEV)
    L = torch.as_tensor(rng.integers(2, T + 1, size=B).astype(np.int32), device=DEV)
    H = torch.randn((B, T, d), device=DEV).to(torch.bfloat16)
    A = torch.rand((B, T, R), device=DEV).to(torch.bfloat16).transpose(1, 2)      # key-major
    A_host = torch.empty_strided(A.shape, A.stride(), dtype=A.dtype, pin_memory=True)
    A_host.copy_(A)
    out = []
    for src in (A, A_host, A.contiguous()):                                      # ... and head-major
        index = torch.empty(pk.pldp_index_size(B, V), dtype=torch.uint8, device=DEV)
        pk.pldp_index_build(ids, L, V, index)
        buf = Buffers(B, K, V, 64, DEV)
        pk.pldp_draft_step(ids, L, 1, 3, buf.cand, buf.cnt, buf.ml, K, buf.draft, buf.dlen, None, H=H,
                           best_h=buf.best_h, A=src, best_a=buf.best_a, a_scores=buf.scores_a,
                           best_a_score=buf.bscore_a, draft_from="attention", status=buf.status, index=index, V=V)
        out.append(snapshot(buf))
    for k in ("cand", "cnt", "best_h", "best_a", "scores_a", "bscore_a", "draft", "dlen", "status"):
        assert np.array_equal(out[0][k], out[1][k], equal_nan=True), k
        assert np.array_equal(out[0][k], out[2][k], equal_nan=True), k
    assert (out[0]["cnt"] > 0).sum() > B // 2
