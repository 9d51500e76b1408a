"""The decode-loop generator on the CPU: its prediction of what greedy verification
will leave (the context lengths, from which it writes the attention rows of the next
query) equals the oracle's verification of the same drafts on the same planted logits,
including clamped draft lengths and a context that runs out of capacity."""
import numpy as np
import torch

import oracle
import workloads as wl
from tests._parity import host


def test_next_lengths_match_oracle_verification():
    w = wl.CONFIGS["decode_loop_b128_ctx32k"].replace(B=6, prompt_len=192, out_len=64, V=100, d=16, layers=1, heads=4,
                                 planted_heads=2)
    loop = wl.DecodeLoop(w, steps=6, device="cpu")
    K, T_cap = w.K, loop.T_cap
    rng = np.random.default_rng(5)
    for s in range(4):
        if s == 2:
            loop.seq_len[0] = T_cap - 2                       # little room left: CAPACITY for n >= 2
        loop.step_inputs(s)
        L = loop.seq_len.long()
        pos = (L[:, None] + torch.arange(K)[None]).clamp(max=T_cap - 1)
        draft = loop.gt.gather(1, pos).to(torch.int32)       # the drafts greedy decoding accepts whole ...
        for b in range(w.B):                                  # ... then a mismatch at a random place or none
            j = int(rng.integers(0, K + 1))
            if j < K:
                draft[b, j] = (int(draft[b, j]) + 1) % w.V
        dlen = torch.as_tensor(rng.integers(0, K + 1, size=w.B), dtype=torch.int32)
        dlen[1], dlen[2] = K + 3, -2                          # clamped into [0, K]
        pred = loop.next_lengths(draft, dlen).numpy()
        L_o = host(loop.seq_len).copy()
        o = oracle.verify_greedy(host(loop.logits), host(draft), host(dlen), seq_len=L_o, T_cap=T_cap)
        assert np.array_equal(pred, L_o), (s, pred, L_o, o["accept_len"])
        loop.seq_len.copy_(torch.as_tensor(L_o))              # advance as the verification would
