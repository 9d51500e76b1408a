"""Pins the oracle to hand-worked cases (tests/golden/*.txt).

Each fixture line was worked out by hand from the paper's definitions (Eq. 1-3,
Sec. 4.3, Sec. 4.4); none was produced by a program.
"""
import math
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _lines(name):
    with open(os.path.join(GOLDEN, name)) as f:
        for ln in f:
            ln = ln.strip()
            if ln and not ln.startswith("#"):
                yield [p.strip() for p in ln.split("|")]


def _ints(s):
    return [] if s == "-" else [int(v) for v in s.split()]


def _floats(s):
    return [float(v) for v in s.split()]


FIND = list(_lines("find_candidates.txt"))


@pytest.mark.parametrize("case", FIND, ids=[f"find{i}" for i in range(len(FIND))])
def test_find_candidates_golden(orc, case):
    ids, L, nmin, nmax, ccap, exp_pos, exp_cnt, exp_ml, exp_st = case
    ids = np.array([_ints(ids)], np.int32)
    cand, cnt, ml, st = orc.find_candidates(ids, [int(L)], int(nmin), int(nmax), int(ccap))
    exp_pos = _ints(exp_pos)
    assert int(cnt[0]) == int(exp_cnt)
    assert int(ml[0]) == int(exp_ml)
    assert int(st[0]) == int(exp_st)
    assert cand[0, :len(exp_pos)].tolist() == exp_pos


HID_ROWS = np.array([[1, 2, 3, 4], [-1, -2, -3, -4], [2, 4, 6, 8], [4, -2, 0, 0],
                     [0, 0, 0, 0], [1, 0, 0, 0], [1, 2, 3, 4], [7, 7, 7, 7]], np.float32)
ATT_ROWS = np.array([[2, 3, 6, 0, 6, 0], [8, 1, 1, 3, 2, 0], [0, 9, 2, 1, 1, 0]], np.float32) / 16

RANK = list(_lines("rank.txt"))


def _score_eq(got, want):
    if math.isinf(want):
        return math.isinf(got) and (got > 0) == (want > 0)
    return abs(got - want) <= 1e-15


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("case", RANK, ids=[f"rank{i}" for i in range(len(RANK))])
def test_rank_golden(orc, case, dtype):
    conv = (lambda a: a) if dtype == "f32" else orc.bf16_bits   # every value is exact in bf16
    if case[0] == "hidden":
        _, thr, cands, exp_scores, exp_best = case
        cands = _ints(cands)
        H = conv(HID_ROWS[None])
        scores, best, _ = orc.rank_hidden(H, [8], np.array([cands], np.int32), [len(cands)],
                                          threshold=float(thr))
        want = _floats(exp_scores)
    else:
        _, agg, rows, cands, exp_scores, exp_best = case
        cands = _ints(cands)
        A = conv(ATT_ROWS[None])
        row_idx = None if rows == "-" else _ints(rows)
        scores, best, _ = orc.rank_attention(A, [6], np.array([cands], np.int32), [len(cands)],
                                             row_idx=row_idx,
                                             agg=orc.AGG_MAX if agg == "max" else orc.AGG_SUM)
        want = [v / 16 for v in _floats(exp_scores)]
    assert all(_score_eq(g, w) for g, w in zip(scores[0, :len(cands)].tolist(), want)), scores
    assert int(best[0]) == int(exp_best)


DV = list(_lines("draft_verify.txt"))


@pytest.mark.parametrize("case", DV, ids=[f"dv{i}" for i in range(len(DV))])
def test_draft_verify_golden(orc, case):
    if case[0] == "draft":
        _, ids, L, best, K, exp_draft, exp_len = case
        draft, dl = orc.extract_draft(np.array([_ints(ids)], np.int32), [int(L)], [int(best)], int(K))
        assert draft[0].tolist() == _ints(exp_draft)
        assert int(dl[0]) == int(exp_len)
        return
    (_, rows, draft, dlen, ids, L, exp_arg, exp_acc, exp_next, exp_ids, exp_L, exp_kv,
     exp_st) = case
    logits = np.array([_floats(r) for r in rows.split(";")], np.float32)[None]
    for conv in (lambda a: a, orc.bf16_bits):
        ids_a = np.array([_ints(ids)], np.int32)
        L_a = np.array([int(L)], np.int32)
        out = orc.verify_greedy(conv(logits), np.array([_ints(draft)], np.int32), [int(dlen)],
                                ids=ids_a, seq_len=L_a, kv_keep=True)
        assert out["argmax"][0].tolist() == _ints(exp_arg)
        assert int(out["accept_len"][0]) == int(exp_acc)
        assert int(out["next_token"][0]) == int(exp_next)
        assert ids_a[0].tolist() == _ints(exp_ids)
        assert int(L_a[0]) == int(exp_L)
        assert int(out["kv_keep_len"][0]) == int(exp_kv)
        assert int(out["status"][0]) == int(exp_st)
