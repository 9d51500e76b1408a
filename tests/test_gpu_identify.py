"""GPU parity of induction-head identification (Sec. 4.2.1): pldp_identify_heads
and pldp_top_heads against the oracle.  Every decision here is exact (integer
overlaps, comparisons of exactly widened values), so counts and r* are compared
bit for bit."""
import numpy as np
import pytest
import torch

import oracle
import workloads as wl
from tests._parity import host

pytestmark = pytest.mark.gpu
DEV = "cuda"


def i32(x):
    return torch.as_tensor(np.asarray(x, np.int32), device=DEV)


# T divisible by 8 (bf16) / 4 (f32) takes 16-byte loads; 301 takes element loads
@pytest.mark.parametrize("T,dtype", [(256, torch.bfloat16), (301, torch.bfloat16), (200, torch.float32),
                                     (4096, torch.bfloat16)])
@pytest.mark.parametrize("V,max_suffix", [(3, 64), (20, 2), (200, 64)])
# R = 5: one CTA per observation (a cluster of one); R = 20: 3 CTAs of 8 rows per
# observation, one cluster of 3; R = 72: 9 CTAs in clusters of 8, the grid padded with 7
# CTAs that hold no rows but take part in the scan
@pytest.mark.parametrize("R", [5, 20, 72])
def test_identify_heads_matches_oracle(lib, T, dtype, V, max_suffix, R):
    rng = np.random.default_rng(T + V + max_suffix + R)
    B = 24
    ids = rng.integers(0, V, size=(B, T)).astype(np.int32)
    pos = rng.integers(1, T, size=B).astype(np.int32)
    pos[0], pos[1] = 0, T                                          # invalid: SEQ_LEN
    A = torch.from_numpy(rng.integers(0, 5, size=(B, R, T)).astype(np.float32)).to(dtype)   # ties
    for b in range(2, B, 2):                                        # some rows peak at a repeat
        p = pos[b]
        occ = np.nonzero(ids[b, :p] == ids[b, p])[0]
        if occ.size:
            A[b, rng.integers(0, R), occ[-1]] = 9.0
    A = A.to(DEV)
    counts = torch.full((R,), 3, dtype=torch.int32, device=DEV)   # added to
    rs = torch.full((B,), -7, dtype=torch.int32, device=DEV)
    st = torch.zeros(B, dtype=torch.int32, device=DEV)
    lib.pldp_identify_heads(i32(ids), i32(pos), A, counts, max_suffix=max_suffix, r_star=rs, status=st)
    oc, ors, ost = oracle.identify_heads(ids, pos, host(A), max_suffix, counts=np.full(R, 3, np.uint32))
    assert np.array_equal(host(rs), ors)
    assert np.array_equal(host(counts).view(np.uint32), oc)
    assert np.array_equal(host(st).view(np.uint32), ost)


def test_identify_recovers_planted_heads(lib):
    w = wl.CONFIGS["attention_b32_ctx8k"].replace(B=32, prompt_len=3000, out_len=1000, V=8000,
                                                  attn_layout="head")   # identification reads whole rows
    tok, src = wl.token_streams(w, w.T, 99)
    rng = np.random.default_rng(100)
    obs_b, obs_p = [], []
    for b in range(w.B):
        inside = [p for p in range(w.prompt_len + 2, w.T)
                  if src[b, p] >= 2 and src[b, p - 1] == src[b, p] - 1 and src[b, p - 2] == src[b, p] - 2]
        for p in rng.choice(inside, size=min(4, len(inside)), replace=False):
            obs_b.append(b)
            obs_p.append(int(p))
    n = len(obs_b)
    ids = i32(tok[obs_b])
    pos = i32(obs_p)
    seq_len = torch.tensor([p + 1 for p in obs_p], dtype=torch.int32, device=DEV)   # x_t = x_p, query p-1
    src_last = torch.tensor([src[b, p] for b, p in zip(obs_b, obs_p)], dtype=torch.int32, device=DEV)
    gen = torch.Generator(device=DEV).manual_seed(101)
    A = wl.gen_attention(w.replace(B=n), seq_len, src_last, w.T, DEV, gen)
    counts = torch.zeros(w.R, dtype=torch.int32, device=DEV)
    rs = torch.zeros(n, dtype=torch.int32, device=DEV)
    lib.pldp_identify_heads(ids, pos, A, counts, r_star=rs)
    assert np.array_equal(host(rs), host(src_last))
    oc, _, _ = oracle.identify_heads(host(ids), host(pos), host(A))
    assert np.array_equal(host(counts).view(np.uint32), oc)
    planted = wl.induction_rows(w)
    top = torch.zeros(planted.size, dtype=torch.int32, device=DEV)
    lib.pldp_top_heads(counts, planted.size, top)
    assert sorted(host(top).tolist()) == sorted(planted.tolist())


@pytest.mark.parametrize("R,k", [(1, 1), (37, 5), (128, 32), (8192, 50)])
def test_top_heads_matches_stable_sort(lib, R, k):
    rng = np.random.default_rng(R + k)
    c = rng.integers(0, 6, size=R).astype(np.int32)               # many ties
    out = torch.full((k,), -1, dtype=torch.int32, device=DEV)
    lib.pldp_top_heads(i32(c), k, out)
    want = np.argsort(-c.astype(np.int64), kind="stable")[:k]
    assert np.array_equal(host(out), want)
