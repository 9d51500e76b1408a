"""The Python binding refuses mis-sized buffers before it calls the library:
every case below raises ValueError on the host, and nothing is launched."""
import pytest
import torch

from tests._parity import Buffers

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _i32(*shape):
    return torch.zeros(shape, dtype=torch.int32, device=DEV)


def test_short_outputs_are_refused(lib):
    B, T, C, K, V = 4, 64, 8, 3, 50
    ids, L = _i32(B, T), torch.full((B,), 10, dtype=torch.int32, device=DEV)
    buf = Buffers(B, K, V, C, DEV)
    with pytest.raises(ValueError, match="seq_len"):
        lib.pldp_find_candidates(ids, L[:B - 1], 1, 3, buf.cand, buf.cnt, buf.ml)
    with pytest.raises(ValueError, match="match_len"):
        lib.pldp_find_candidates(ids, L, 1, 3, buf.cand, buf.cnt, buf.ml[:2])
    with pytest.raises(ValueError, match="status"):
        lib.pldp_find_candidates(ids, L, 1, 3, buf.cand, buf.cnt, buf.ml,
                                 status=torch.zeros(B, dtype=torch.int64, device=DEV))
    H = torch.zeros((B, T, 32), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(ValueError, match="scores"):
        lib.pldp_rank_hidden(H, L, buf.cand, buf.cnt, buf.best_h, scores=buf.scores_h[:, :C - 1].contiguous())
    logits = torch.zeros((B, K + 1, V), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(ValueError, match="argmax"):
        lib.pldp_verify_greedy(logits, buf.draft, buf.dlen, buf.acc, buf.nxt, buf.ws, argmax=buf.argmax[:, :K])
    with pytest.raises(ValueError, match="rows"):
        lib.pldp_verify_greedy(logits, buf.draft, buf.dlen, buf.acc, buf.nxt, buf.ws, ids=ids[:B - 1], seq_len=L)
    with pytest.raises(ValueError, match="T_cap"):
        lib.pldp_extract_draft(ids, L, buf.best_h, buf.draft, buf.dlen, T_cap=T + 1)


def test_short_model_artifacts_are_refused(lib):
    B, T, C, K, V = 4, 64, 8, 3, 50
    ids, L = _i32(B, T), torch.full((B,), 10, dtype=torch.int32, device=DEV)
    buf = Buffers(B, K, V, C, DEV)
    H = torch.zeros((B, T - 1, 32), dtype=torch.bfloat16, device=DEV)      # one position short
    A = torch.zeros((B - 1, 2, T), dtype=torch.bfloat16, device=DEV)       # one sequence short
    with pytest.raises(ValueError, match="H must cover"):
        lib.pldp_draft_step(ids, L, 1, 3, buf.cand, buf.cnt, buf.ml, K, buf.draft, buf.dlen, buf.dws,
                            H=H, best_h=buf.best_h)
    with pytest.raises(ValueError, match="A must cover"):
        lib.pldp_draft_step(ids, L, 1, 3, buf.cand, buf.cnt, buf.ml, K, buf.draft, buf.dlen, buf.dws,
                            A=A, best_a=buf.best_a, draft_from="attention")
    logits = torch.zeros((B, K + 1, V), dtype=torch.bfloat16, device=DEV)
    ix = torch.zeros(lib.pldp_index_size(B + 1, V), dtype=torch.uint8, device=DEV)
    with pytest.raises(ValueError, match="ids must be"):                   # one more context than logits
        lib.pldp_verify_greedy_draft(logits, buf.draft, buf.dlen, buf.acc, buf.nxt, buf.ws, _i32(B + 1, T),
                                     torch.full((B + 1,), 10, dtype=torch.int32, device=DEV), 1, 3,
                                     buf.cand, buf.cnt, buf.ml, buf.draft, buf.dlen, ix)
