"""Pins the oracle to things other than itself (CPU only).

* Candidate search (Eq. 1 + longest-suffix n-gram): an independent brute force
  that finds n-gram occurrences with ``bytes.find`` over a fixed-width byte
  encoding of the tokens, run exhaustively on tiny contexts.
* Hidden ranking (Eq. 3): ``scipy.spatial.distance.cosine`` on random rows, and
  the planted-source statistic (source + N(0, 0.1^2) noise has cosine
  1/sqrt(1.01) ~ 0.995; unrelated N(0,1) rows have |cos| < 0.1 at d = 4096).
* Attention ranking (Eq. 2): ``numpy`` max/sum over the selected rows.
* Verification (Sec. 4.4): ``numpy.argmax`` (documented first occurrence) and
  the accept-length invariants.
* Sampling verification (Sec. 4.4 at T > 0): ``scipy.special.softmax`` and
  ``numpy.searchsorted`` over a grid of uniforms (inverse-CDF sampling), the
  low-temperature limit (argmax), equal logits (floor(u V)), zero-probability
  tokens, and the acceptance rate p(draft token) that makes the step lossless.
"""
import itertools

import numpy as np
import pytest
from scipy.spatial.distance import cosine as scipy_cosine
from scipy.special import softmax as scipy_softmax


# ----------------------------------------------------------------------------
# candidate search
# ----------------------------------------------------------------------------
def _occurrences_by_bytes(seq, L, nmin, nmax):
    """Longest-suffix n-gram occurrences, found by substring search on bytes."""
    t = L - 1
    if t < 1:
        return [], 0
    enc = b"".join(int(v).to_bytes(4, "big", signed=True) for v in seq[:L])
    for n in range(nmax, nmin - 1, -1):
        if t - n + 1 < 0:
            continue
        needle = enc[4 * (t - n + 1): 4 * (t + 1)]
        hay = enc[: 4 * t]            # the n-gram must END before t, i.e. j < t
        found, start = [], 0
        while True:
            k = hay.find(needle, start)
            if k < 0:
                break
            if k % 4 == 0:            # token-aligned hit; it ends at position j
                found.append(k // 4 + n - 1)
            start = k + 1
        if found:
            return sorted(found), n
    return [], 0


def test_find_exhaustive_binary_alphabet(orc):
    # every binary context of length 1..9 (1022 contexts), several n ranges
    ctx, lens = [], []
    for L in range(1, 10):
        for bits in itertools.product([0, 1], repeat=L):
            ctx.append(list(bits) + [0] * (9 - L))
            lens.append(L)
    ids = np.array(ctx, np.int32)
    for nmin, nmax in [(1, 1), (1, 2), (1, 3), (2, 3), (3, 3), (1, 4)]:
        cand, cnt, ml, st = orc.find_candidates(ids, lens, nmin, nmax, 16)
        for b, L in enumerate(lens):
            want, n = _occurrences_by_bytes(ids[b], L, nmin, nmax)
            assert cnt[b] == len(want) and ml[b] == n, (ids[b, :L], nmin, nmax)
            assert cand[b, :len(want)].tolist() == want
            assert st[b] == 0


@pytest.mark.parametrize("V,T", [(3, 40), (5, 200), (50, 300)])
def test_find_random_vs_bytes_search(orc, V, T):
    rng = np.random.default_rng(V * 1000 + T)
    B = 64
    ids = rng.integers(0, V, size=(B, T)).astype(np.int32)
    lens = rng.integers(0, T + 1, size=B)
    cand, cnt, ml, st = orc.find_candidates(ids, lens, 1, 3, T)
    for b in range(B):
        want, n = _occurrences_by_bytes(ids[b], lens[b], 1, 3)
        assert cnt[b] == len(want) and ml[b] == n
        assert cand[b, :len(want)].tolist() == want


def test_find_unigram_is_eq1(orc):
    rng = np.random.default_rng(7)
    ids = rng.integers(0, 6, size=(32, 50)).astype(np.int32)
    lens = rng.integers(2, 51, size=32)
    cand, cnt, ml, _ = orc.find_candidates(ids, lens, 1, 1, 50)
    for b in range(32):
        t = lens[b] - 1
        eq1 = [j for j in range(t) if ids[b, j] == ids[b, t]]        # Eq. 1 literally
        assert cand[b, :cnt[b]].tolist() == eq1
        assert ml[b] == (1 if eq1 else 0)


def test_find_overflow_keeps_first_ascending(orc):
    ids = np.zeros((1, 100), np.int32)
    cand, cnt, ml, st = orc.find_candidates(ids, [100], 1, 3, 10)
    assert cnt[0] == 97 and ml[0] == 3            # j = 2..98
    assert cand[0].tolist() == list(range(2, 12))
    assert st[0] == orc.ST_CAND_OVERFLOW


# ----------------------------------------------------------------------------
# hidden-state ranking
# ----------------------------------------------------------------------------
def test_rank_hidden_matches_scipy(orc):
    rng = np.random.default_rng(11)
    B, T, d = 4, 30, 257
    H = rng.standard_normal((B, T, d)).astype(np.float32)
    lens = np.array([30, 17, 5, 30], np.int32)
    cands = np.tile(np.arange(0, 29, dtype=np.int32), (B, 1))
    cnt = np.array([29, 16, 4, 29], np.int32)
    scores, best, bs = orc.rank_hidden(H, lens, cands, cnt)
    for b in range(B):
        t = lens[b] - 1
        ref = [-np.inf] + [1.0 - scipy_cosine(H[b, j - 1].astype(np.float64),
                                              H[b, t - 1].astype(np.float64)) for j in range(1, cnt[b])]
        np.testing.assert_allclose(scores[b, :cnt[b]], ref, rtol=0, atol=1e-12)
        jb = int(np.argmax(ref))
        assert best[b] == jb and abs(bs[b] - ref[jb]) < 1e-12


def test_rank_hidden_bf16_is_exact_widening(orc):
    rng = np.random.default_rng(12)
    H32 = rng.standard_normal((2, 20, 64)).astype(np.float32)
    bits = orc.bf16_bits(H32)
    exact = orc.bf16_to_f32(bits)
    cands = np.tile(np.arange(1, 19, dtype=np.int32), (2, 1))
    s_bf, b_bf, _ = orc.rank_hidden(bits, [20, 20], cands, [18, 18])
    s_32, b_32, _ = orc.rank_hidden(exact, [20, 20], cands, [18, 18])
    assert np.array_equal(s_bf, s_32) and np.array_equal(b_bf, b_32)


def test_rank_hidden_planted_source_wins(orc):
    """Sec. 4.2.2 premise: the row before the true copy source resembles the query row.
    Query H_{t-1} = H_{s-1} + N(0, 0.1^2); the source s must win, with the
    expected cosine ~ 1/sqrt(1.01); wrong query/candidate rows would not."""
    rng = np.random.default_rng(13)
    B, T, d = 8, 64, 4096
    H = rng.standard_normal((B, T, d)).astype(np.float32)
    lens = np.full(B, T, np.int32)
    t = T - 1
    srcs = rng.integers(1, t - 2, size=B)
    for b in range(B):
        H[b, t - 1] = H[b, srcs[b] - 1] + 0.1 * rng.standard_normal(d).astype(np.float32)
    cands = np.tile(np.arange(1, t, dtype=np.int32), (B, 1))
    scores, best, bs = orc.rank_hidden(H, lens, cands, np.full(B, t - 1, np.int32))
    assert best.tolist() == srcs.tolist()
    assert np.all(np.abs(bs - 1 / np.sqrt(1.01)) < 0.005)
    others = np.array([[scores[b, i] for i in range(t - 1) if i + 1 != srcs[b] and i + 2 != t]
                       for b in range(B)])
    assert np.abs(others).max() < 0.1


def test_rank_hidden_zero_norm_threshold_ineligible(orc):
    H = np.zeros((1, 6, 8), np.float32)
    H[0, 4] = 1.0                                   # query row H_{t-1}, t = 5
    H[0, 2] = -1.0
    cands = np.array([[0, 1, 3]], np.int32)         # j=0 ineligible, j=1 -> H_0 = 0, j=3 -> H_2
    scores, best, bs = orc.rank_hidden(H, [6], cands, [3])
    assert scores[0, 0] == -np.inf and scores[0, 1] == 0.0 and scores[0, 2] == -1.0
    assert best[0] == 1 and bs[0] == 0.0
    _, best, bs = orc.rank_hidden(H, [6], cands, [3], threshold=0.0)     # strict: 0 > 0 fails
    assert best[0] == -1 and bs[0] == -np.inf


# ----------------------------------------------------------------------------
# attention ranking
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("agg", ["max", "sum"])
def test_rank_attention_matches_numpy(orc, agg):
    rng = np.random.default_rng(21)
    B, R, T = 5, 12, 40
    A = rng.random((B, R, T)).astype(np.float32)
    lens = rng.integers(2, T + 1, size=B).astype(np.int32)
    C = 16
    cands = np.stack([np.sort(rng.choice(T, C, replace=False)) for _ in range(B)]).astype(np.int32)
    cnt = rng.integers(0, C + 1, size=B).astype(np.int32)
    rows = np.array([3, 0, 7, 11], np.int32)
    code = orc.AGG_MAX if agg == "max" else orc.AGG_SUM
    scores, best, bs = orc.rank_attention(A, lens, cands, cnt, row_idx=rows, agg=code)
    for b in range(B):
        sel = A[b][rows].astype(np.float64)
        red = sel.max(axis=0) if agg == "max" else sel.sum(axis=0)
        want = [red[j] if j < lens[b] - 1 else -np.inf for j in cands[b, :cnt[b]]]
        np.testing.assert_allclose(scores[b, :cnt[b]], want, rtol=0, atol=1e-12)
        valid = [(w, -j) for w, j in zip(want, cands[b, :cnt[b]]) if np.isfinite(w)]
        assert best[b] == (-max(valid)[1] if valid else -1)


def test_rank_attention_planted_key_is_candidate_itself(orc):
    """Reading of Eq. 2: the induction row of query t-1 peaks at key j (the copied
    token), so planting mass at key s selects s, not s+1 or s-1."""
    rng = np.random.default_rng(22)
    B, R, T = 6, 8, 50
    logits = rng.standard_normal((B, R, T))
    srcs = rng.integers(5, 40, size=B)
    for b in range(B):
        logits[b, :3, srcs[b]] += 6.0
    A = np.exp(logits) / np.exp(logits).sum(-1, keepdims=True)
    cands = np.tile(np.arange(0, T - 1, dtype=np.int32), (B, 1))
    _, best, _ = orc.rank_attention(A.astype(np.float32), np.full(B, T, np.int32), cands,
                                    np.full(B, T - 1, np.int32))
    assert best.tolist() == srcs.tolist()


# ----------------------------------------------------------------------------
# draft + verify
# ----------------------------------------------------------------------------
def test_extract_draft_is_following_span(orc):
    rng = np.random.default_rng(31)
    B, T, K = 40, 30, 7
    ids = rng.integers(0, 1000, size=(B, T)).astype(np.int32)
    lens = rng.integers(0, T + 1, size=B).astype(np.int32)
    best = rng.integers(-1, T, size=B).astype(np.int32)
    draft, dl = orc.extract_draft(ids, lens, best, K)
    for b in range(B):
        t = lens[b] - 1
        span = list(ids[b, best[b] + 1: t + 1][:K]) if 0 <= best[b] < t else []
        assert dl[b] == len(span)
        assert draft[b].tolist() == span + [-1] * (K - len(span))


@pytest.mark.parametrize("bf16", [False, True])
def test_verify_matches_numpy_argmax_and_invariants(orc, bf16):
    rng = np.random.default_rng(41 + bf16)
    B, K, V = 64, 6, 37
    logits = rng.integers(-3, 4, size=(B, K + 1, V)).astype(np.float32)   # many exact ties
    logits[logits == 0] = np.where(rng.random((logits == 0).sum()) < 0.5, -0.0, 0.0)
    am = logits.argmax(-1)                                                 # first occurrence
    draft = np.where(rng.random((B, K)) < 0.8, am[:, :K], rng.integers(0, V, size=(B, K)))
    dlen = rng.integers(0, K + 1, size=B)
    draft = np.where(np.arange(K)[None] < dlen[:, None], draft, -1).astype(np.int32)
    T_cap = 20
    ids = rng.integers(0, V, size=(B, T_cap)).astype(np.int32)
    lens = rng.integers(1, T_cap + 1, size=B).astype(np.int32)
    ids0, lens0 = ids.copy(), lens.copy()
    x = orc.bf16_bits(logits) if bf16 else logits
    out = orc.verify_greedy(x, draft, dlen, ids=ids, seq_len=lens, kv_keep=True)
    assert np.array_equal(out["argmax"], am)
    for b in range(B):
        d = dlen[b]
        mism = [i for i in range(d) if draft[b, i] != am[b, i]]
        n = mism[0] if mism else d
        assert 0 <= out["accept_len"][b] <= d <= K
        assert out["accept_len"][b] == n and out["next_token"][b] == am[b, n]
        assert out["kv_keep_len"][b] == lens0[b] + n
        if lens0[b] + n + 1 <= T_cap:
            assert lens[b] == lens0[b] + n + 1 and out["status"][b] == 0
            emitted = list(draft[b, :n]) + [am[b, n]]
            assert ids[b, lens0[b]:lens[b]].tolist() == emitted
            assert np.array_equal(ids[b, :lens0[b]], ids0[b, :lens0[b]])
        else:
            assert lens[b] == lens0[b] and out["status"][b] == orc.ST_CAPACITY
            assert np.array_equal(ids[b], ids0[b])


# ----------------------------------------------------------------------------
# sampling verification
# ----------------------------------------------------------------------------
def _grid_draws(orc, logits_row, T, us):
    """Draws of the oracle for one logits row under each uniform in ``us``
    (one sequence per uniform, K = 1; row 1 gets the uniform reversed)."""
    N, V = len(us), logits_row.size
    logits = np.broadcast_to(logits_row.astype(np.float32), (N, 2, V)).copy()
    u = np.stack([us, us[::-1]], axis=1).astype(np.float32)
    out = orc.verify_sample(logits, u, np.zeros((N, 1), np.int32), np.zeros(N, np.int32), temperature=T)
    return out["sampled"][:, 0], out["sampled"][:, 1][::-1]


@pytest.mark.parametrize("T", [1.0, 0.5, 2.0])
def test_sample_is_inverse_cdf_of_softmax(orc, T):
    rng = np.random.default_rng(int(T * 10))
    row = rng.normal(0, 1.5, size=7).astype(np.float32)
    cdf = np.cumsum(scipy_softmax(row.astype(np.float64) / T))
    us = ((np.arange(4000) + 0.5) / 4000).astype(np.float32)
    keep = np.min(np.abs(us.astype(np.float64)[:, None] - cdf[None, :]), axis=1) > 1e-9
    want = np.searchsorted(cdf, us.astype(np.float64), side="right")   # smallest v with cdf_v > u
    got0, got1 = _grid_draws(orc, row, T, us)
    assert np.array_equal(got0[keep], want[keep]) and np.array_equal(got1[keep], want[keep])
    # the frequencies over the grid are the probabilities
    freq = np.bincount(got0, minlength=7) / us.size
    assert np.allclose(freq, np.diff(np.concatenate([[0.0], cdf])), atol=1.0 / us.size)


def test_sample_hand_worked(orc):
    # logits ln 1, ln 2, ln 3 at T = 1: p = 1/6, 2/6, 3/6, cumulative 1/6, 1/2, 1
    row = np.log(np.array([1.0, 2.0, 3.0])).astype(np.float32)
    us = np.array([0.0, 0.1, 0.17, 0.3, 0.49, 0.51, 0.99], np.float32)
    got, _ = _grid_draws(orc, row, 1.0, us)
    assert got.tolist() == [0, 0, 1, 1, 1, 2, 2]


def test_sample_low_temperature_is_argmax(orc):
    rng = np.random.default_rng(5)
    row = (rng.permutation(40) * 0.05).astype(np.float32)            # distinct, gaps >= 0.05
    us = np.linspace(1e-6, 0.999, 300).astype(np.float32)       # u = 0 draws the first p > 0
    got, _ = _grid_draws(orc, row, 1e-3, us)
    assert (got == np.argmax(row)).all()


def test_sample_equal_logits_is_floor_uV(orc):
    V = 12
    us = ((np.arange(600) + 0.25) / 600).astype(np.float32)
    got, _ = _grid_draws(orc, np.full(V, 0.7, np.float32), 1.0, us)
    want = np.floor(us.astype(np.float64) * V).astype(int)
    near = np.abs(us.astype(np.float64) * V - np.round(us.astype(np.float64) * V)) < 1e-6
    assert np.array_equal(got[~near], want[~near])


def test_sample_never_draws_zero_probability(orc):
    row = np.array([-1000.0, 0.0, -1000.0, 0.5, -1000.0], np.float32)
    us = np.array([0.0, 1e-12, 0.3, 0.999999], np.float32)
    got, _ = _grid_draws(orc, row, 1.0, us)
    assert set(got.tolist()) <= {1, 3} and got[0] == 1


def test_sample_acceptance_rate_is_p_of_draft(orc):
    """The draft token is accepted exactly when the draw equals it, so over a grid of
    uniforms the accepted fraction is p(draft); on a rejection the bonus is the draw
    (never the draft token), and with every position accepted the bonus is the draw
    at position K."""
    row = np.array([0.3, -0.2, 1.1, 0.0], np.float32)
    p = scipy_softmax(row.astype(np.float64))
    N = 5000
    us = ((np.arange(N) + 0.5) / N).astype(np.float32)
    for tok in range(4):
        logits = np.broadcast_to(row, (N, 2, 4)).copy()
        u = np.stack([us, us[::-1]], axis=1)
        draft = np.full((N, 1), tok, np.int32)
        out = orc.verify_sample(logits, u, draft, np.ones(N, np.int32))
        acc = out["accept_len"]
        assert abs(acc.mean() - p[tok]) <= 2.0 / N
        rej = acc == 0
        assert (out["next_token"][rej] != tok).all()
        assert np.array_equal(out["next_token"][rej], out["sampled"][rej, 0])
        assert np.array_equal(out["next_token"][~rej], out["sampled"][~rej, 1])


def test_sample_bookkeeping_matches_greedy_rules(orc):
    rng = np.random.default_rng(77)
    B, K, V, T_cap = 32, 5, 9, 16
    logits = rng.normal(0, 2, size=(B, K + 1, V)).astype(np.float32)
    u = rng.random((B, K + 1)).astype(np.float32)
    first = orc.verify_sample(logits, u, np.zeros((B, K), np.int32), np.zeros(B, np.int32))
    y = first["sampled"]
    draft = np.where(rng.random((B, K)) < 0.7, y[:, :K], rng.integers(0, V, size=(B, K))).astype(np.int32)
    dlen = rng.integers(0, K + 1, size=B).astype(np.int32)
    ids = rng.integers(0, V, size=(B, T_cap)).astype(np.int32)
    lens = rng.integers(1, T_cap + 1, size=B).astype(np.int32)
    ids0, lens0 = ids.copy(), lens.copy()
    out = orc.verify_sample(logits, u, draft, dlen, ids=ids, seq_len=lens, kv_keep=True)
    assert np.array_equal(out["sampled"], y)
    for b in range(B):
        mism = [i for i in range(dlen[b]) if draft[b, i] != y[b, i]]
        n = mism[0] if mism else dlen[b]
        assert out["accept_len"][b] == n and out["next_token"][b] == y[b, n]
        assert out["kv_keep_len"][b] == lens0[b] + n
        if lens0[b] + n + 1 <= T_cap:
            assert ids[b, lens0[b]:lens[b]].tolist() == list(draft[b, :n]) + [y[b, n]]
        else:
            assert out["status"][b] == orc.ST_CAPACITY and np.array_equal(ids[b], ids0[b])


# ----------------------------------------------------------------------------
# averaged hidden states (App. B.2)
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("m", [1, 2, 3, 5])
def test_rank_hidden_avg_matches_numpy_window_means(orc, m):
    rng = np.random.default_rng(300 + m)
    B, T, d, C = 4, 24, 16, 8
    H = rng.normal(size=(B, T, d)).astype(np.float32)
    lens = np.array([T, 13, 3, 2], np.int32)
    cand = np.zeros((B, C), np.int32)
    cnt = np.zeros(B, np.int32)
    for b in range(B):
        js = np.unique(rng.integers(0, max(lens[b] - 1, 1), size=6))
        js = js[js < max(lens[b] - 1, 1)]
        cnt[b] = js.size
        cand[b, :js.size] = js
    s, best, bs = orc.rank_hidden_avg(H, lens, cand, cnt, m)
    for b in range(B):
        t = lens[b] - 1
        def mean(p):
            return H[b, max(0, p - m + 1):p + 1].astype(np.float64).mean(axis=0)
        want = []
        for i in range(cnt[b]):
            j = cand[b, i]
            want.append(1.0 - scipy_cosine(mean(j - 1), mean(t - 1)) if 1 <= j < t else -np.inf)
        assert np.allclose(s[b, :cnt[b]], want, atol=1e-12, rtol=0)
        ok = [(w, -cand[b, i]) for i, w in enumerate(want) if np.isfinite(w)]
        assert best[b] == (-max(ok)[1] if ok else -1)


def test_rank_hidden_avg_m1_is_eq3_exactly(orc):
    rng = np.random.default_rng(17)
    B, T, d, C = 3, 40, 32, 10
    H = rng.normal(size=(B, T, d)).astype(np.float32)
    lens = np.array([40, 22, 5], np.int32)
    cand = np.tile(np.arange(0, 2 * C, 2, dtype=np.int32), (B, 1))
    cnt = np.array([10, 10, 3], np.int32)
    a = orc.rank_hidden_avg(H, lens, cand, cnt, 1, threshold=0.05)
    e = orc.rank_hidden(H, lens, cand, cnt, threshold=0.05)
    assert np.array_equal(a[0], e[0], equal_nan=True) and np.array_equal(a[1], e[1])


def test_rank_hidden_avg_tie_goes_to_smaller_position(orc):
    # candidates 9 and 17 have identical windows (rows 6..8 copied to 14..16): equal scores
    rng = np.random.default_rng(23)
    H = rng.normal(size=(1, 30, 8)).astype(np.float32)
    H[0, 14:17] = H[0, 6:9]
    cand = np.array([[17, 9, 25]], np.int32)
    s, best, _ = orc.rank_hidden_avg(H, np.array([30], np.int32), cand, np.array([2], np.int32), 3)
    assert s[0, 0] == s[0, 1] and best[0] == 9


# ----------------------------------------------------------------------------
# induction-head identification (Sec. 4.2.1)
# ----------------------------------------------------------------------------
def _identify_brute(ids, pos, A, max_suffix):
    """Direct restatement with Python loops: P, overlap, r* (smallest j on ties),
    and per row numpy's first argmax over keys < p."""
    B, R, _ = A.shape
    counts = np.zeros(R, np.uint32)
    rs = np.full(B, -1, np.int32)
    for b in range(B):
        p = int(pos[b])
        x = ids[b]
        best = (0, 0)
        for j in range(p):
            if x[j] != x[p]:
                continue
            k = 0
            while k < max_suffix and j - k >= 0 and x[j - k] == x[p - k]:
                k += 1
            if (k, -j) > best:
                best = (k, -j)
        if best[0] == 0:
            continue
        rs[b] = -best[1]
        for r in range(R):
            if int(np.argmax(A[b, r, :p])) == rs[b]:
                counts[r] += 1
    return counts, rs


@pytest.mark.parametrize("V,max_suffix", [(2, 64), (3, 2), (5, 1), (50, 64)])
def test_identify_heads_matches_brute_force(orc, V, max_suffix):
    rng = np.random.default_rng(V * 10 + max_suffix)
    B, T, R = 40, 30, 6
    ids = rng.integers(0, V, size=(B, T)).astype(np.int32)
    pos = rng.integers(1, T, size=B).astype(np.int32)
    A = rng.integers(0, 4, size=(B, R, T)).astype(np.float32)       # many equal maxima
    for b in range(0, B, 3):                                       # some rows point at a repeat
        p = pos[b]
        occ = [j for j in range(p) if ids[b, j] == ids[b, p]]
        if occ:
            A[b, rng.integers(0, R), occ[-1]] = 9.0
    c, rs, st = orc.identify_heads(ids, pos, A, max_suffix)
    wc, wrs = _identify_brute(ids, pos, A, max_suffix)
    assert np.array_equal(rs, wrs) and np.array_equal(c, wc) and (st == 0).all()


def test_identify_heads_recovers_planted_heads(orc):
    """Copied spans; rows of 3 planted heads per layer put extra attention on the
    true copy source of the generated token: they are exactly the top heads."""
    import workloads as wl
    w = wl.CONFIGS["attention_b32_ctx8k"].replace(B=24, prompt_len=600, out_len=400, V=5000, layers=2, heads=8,
                                 planted_heads=3)
    tok, src = wl.token_streams(w, w.T, 77)
    rng = np.random.default_rng(78)
    obs_b, obs_p = [], []
    for b in range(w.B):                                           # positions deep inside copied spans
        inside = [p for p in range(w.prompt_len + 2, w.T)
                  if src[b, p] >= 2 and src[b, p - 1] == src[b, p] - 1 and src[b, p - 2] == src[b, p] - 2]
        for p in rng.choice(inside, size=min(4, len(inside)), replace=False):
            obs_b.append(b)
            obs_p.append(p)
    n = len(obs_b)
    ids = tok[obs_b].astype(np.int32)
    pos = np.array(obs_p, np.int32)
    R, T = w.layers * w.heads, w.T
    planted = set(wl.induction_rows(w).tolist())
    logits = rng.normal(size=(n, R, T))
    for i in range(n):
        for r in planted:
            logits[i, r, src[obs_b[i], obs_p[i]]] += 8.0
        logits[i, :, obs_p[i]:] = -np.inf
    A = np.exp(logits - logits.max(-1, keepdims=True))
    A = (A / A.sum(-1, keepdims=True)).astype(np.float32)
    c, rs, _ = orc.identify_heads(ids, pos, A)
    assert np.array_equal(rs, [src[b, p] for b, p in zip(obs_b, obs_p)])
    top = set(np.argsort(-c.astype(np.int64), kind="stable")[:len(planted)].tolist())
    assert top == planted and c[sorted(planted)].min() == n


def test_identify_heads_edges_and_accumulation(orc):
    ids = np.array([[1, 2, 3, 4, 5, 6], [7, 8, 7, 8, 7, 8]], np.int32)
    A = np.zeros((2, 2, 6), np.float32)
    A[1, 0, 3] = 1.0                      # row 0 points at key 3 (x_3 = 8, overlap 4)
    A[1, 1, 1] = 1.0                      # row 1 at key 1 (overlap 2)
    c, rs, st = orc.identify_heads(ids, np.array([5, 5], np.int32), A)
    assert rs.tolist() == [-1, 3] and c.tolist() == [1, 0] and st.tolist() == [0, 0]
    c2, _, _ = orc.identify_heads(ids, np.array([5, 5], np.int32), A, counts=c)
    assert c2.tolist() == [2, 0]
    _, rs, st = orc.identify_heads(ids, np.array([0, 6], np.int32), A)
    assert rs.tolist() == [-1, -1] and st.tolist() == [orc.ST_SEQ_LEN, orc.ST_SEQ_LEN]
