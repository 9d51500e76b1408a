"""The allocation-free verification entry point, for callers that cannot give the
library a workspace (no device allocator of their own, or no cudaMalloc allowed
once serving has started).

It must return exactly what pldp_verify_greedy returns on the same inputs, call
after call, although its scratch is one shared area that outlives every call.
This file is named so that pytest collects it last."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _inputs(seed, B=24, K=12, V=128256, T_cap=96):
    g = torch.Generator(device=DEV).manual_seed(seed)
    logits = torch.randn((B, K + 1, V), generator=g, device=DEV).to(torch.bfloat16)
    am = logits.float().argmax(-1).to(torch.int32)
    keep = torch.rand((B, K), generator=g, device=DEV) < 0.8
    noise = torch.randint(0, V, (B, K), generator=g, device=DEV, dtype=torch.int32)
    draft = torch.where(keep, am[:, :K], noise)
    draft_len = torch.randint(0, K + 1, (B,), generator=g, device=DEV, dtype=torch.int32)
    ids = torch.randint(0, V, (B, T_cap), generator=g, device=DEV, dtype=torch.int32)
    seq_len = torch.randint(1, T_cap - K - 1, (B,), generator=g, device=DEV, dtype=torch.int32)
    return logits, draft, draft_len, ids, seq_len


def _outputs(B, K):
    z = lambda *s: torch.zeros(s, dtype=torch.int32, device=DEV)  # noqa: E731
    return dict(argmax=z(B, K + 1), acc=z(B), nxt=z(B), kv=z(B), status=z(B))


def test_noalloc_matches_workspace_entry_point_twice(lib):
    B, K, V = 24, 12, 128256
    ws = torch.zeros(lib.pldp_verify_workspace_size(B, K, V), dtype=torch.uint8, device=DEV)
    for call, seed in enumerate((11, 12)):          # two calls in a row, different inputs
        logits, draft, dlen, ids, seq_len = _inputs(seed, B, K, V)
        ids_a, len_a, ids_b, len_b = ids.clone(), seq_len.clone(), ids.clone(), seq_len.clone()
        a, b = _outputs(B, K), _outputs(B, K)
        lib.pldp_verify_greedy(logits, draft, dlen, a["acc"], a["nxt"], ws, argmax=a["argmax"],
                               ids=ids_a, seq_len=len_a, kv_keep_len=a["kv"], status=a["status"])
        lib.pldp_verify_greedy_noalloc(logits, draft, dlen, b["acc"], b["nxt"], argmax=b["argmax"],
                                       ids=ids_b, seq_len=len_b, kv_keep_len=b["kv"],
                                       status=b["status"])
        torch.cuda.synchronize()
        for k in a:
            assert torch.equal(a[k], b[k]), (call, k)
        assert torch.equal(ids_a, ids_b) and torch.equal(len_a, len_b), call
        assert int(a["acc"].sum()) > 0                 # the drafts are partly accepted


def test_noalloc_rejects_batches_beyond_its_scratch(lib):
    B, K, V = 20000, 12, 8                             # 20000 * 13 rows of keys > 1 MiB
    assert lib.pldp_verify_workspace_size(B, K, V) > (1 << 20)
    logits = torch.zeros((B, K + 1, V), dtype=torch.bfloat16, device=DEV)
    draft = torch.zeros((B, K), dtype=torch.int32, device=DEV)
    o = _outputs(B, K)
    with pytest.raises(lib.PldpError) as ei:
        lib.pldp_verify_greedy_noalloc(logits, draft, o["acc"], o["acc"], o["nxt"])
    assert ei.value.code == 1 and "scratch" in str(ei.value)
