"""CPU check of the full-size parity tests' host copies: the oracle's rankings on
the sparse host arrays of tests._parity.oracle_rows (only the rows the rankings
read are copied) equal its rankings on the whole tensors."""
import numpy as np
import torch

import oracle
from tests._parity import host, oracle_rows


def test_oracle_rows_hold_what_the_rankings_read():
    rng = np.random.default_rng(5)
    B, T_cap, d, R, V = 7, 60, 24, 6, 4                 # V = 4: many candidates per sequence
    ids = rng.integers(0, V, size=(B, T_cap)).astype(np.int32)
    L = np.array([60, 0, 1, 2, 61, 37, 59], np.int32)   # full, empty, x_t alone, one row, invalid, ragged
    g = torch.Generator().manual_seed(3)
    for dt in (torch.float32, torch.bfloat16):
        H = torch.randn((B, T_cap, d), generator=g).to(dt)
        A = torch.rand((B, R, T_cap), generator=g).to(dt)
        cand, cnt, _, _ = oracle.find_candidates(ids, L, 1, 3, 16)
        assert (cnt[[0, 5, 6]] > 0).all()
        Hs, As = oracle_rows(H, A, L, cand, cnt)
        assert np.count_nonzero(Hs) < Hs.size // 4 and np.count_nonzero(As) < As.size // 4
        for rank, full, sparse in ((oracle.rank_hidden, host(H), Hs), (oracle.rank_attention, host(A), As)):
            s_f, b_f, bs_f = rank(full, L, cand, cnt)
            s_s, b_s, bs_s = rank(sparse, L, cand, cnt)
            assert np.array_equal(s_f, s_s, equal_nan=True)
            assert np.array_equal(b_f, b_s) and np.array_equal(bs_f, bs_s)
