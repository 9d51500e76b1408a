"""CPU oracle of the PLD+ drafting and greedy-verification step (arXiv 2412.01447).

TEST INFRASTRUCTURE ONLY.  The oracle is the independent, slow, obviously
correct reference that the CUDA library is checked against.  Only the test
suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may
import it; the product path (``paper_2412_01447_gb300``) never does, and the two
share no code.

The arithmetic lives in ``pldp_oracle.c`` (plain single-threaded C, fp64).
This module only compiles it with gcc and marshals numpy arrays through ctypes.

Functions and the passages they follow:

* :func:`find_candidates` -- Eq. 1 (Sec. 4.2) with the longest-suffix n-gram rule.
* :func:`rank_hidden`     -- Eq. 3 (Sec. 4.2.2), optional threshold (App. B.3).
* :func:`rank_attention`  -- Eq. 2 (Sec. 4.2.1), max or sum aggregation (Sec. 7.1).
* :func:`extract_draft`   -- Sec. 4.3.
* :func:`verify_greedy`   -- Sec. 4.4 at T = 0 (and Sec. 3: K+1 distributions).

Parity status: every function is pinned by the ``-m "not gpu"`` tests in
``tests/test_oracle_*.py`` (hand-worked golden cases, closed forms, brute force
on tiny inputs, an independent library routine, planted-structure statistics).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pldp_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")

F32, BF16 = 0, 1
AGG_MAX, AGG_SUM = 0, 1
ST_CAND_OVERFLOW, ST_TOKEN_RANGE, ST_CAPACITY, ST_SEQ_LEN, ST_DRAFT_LEN, ST_ROW_INDEX = 1, 2, 4, 8, 16, 32

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``pldp_oracle.c`` into ``liboracle.so`` (gcc -O2, no fast-math)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-Wall",
                               _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB_PATH)
            _configure(lib)
            _lib = lib
    return _lib


def _configure(lib):
    P = ctypes.c_void_p
    i32, i64, dbl = ctypes.c_int, ctypes.c_int64, ctypes.c_double
    lib.pldpo_find_candidates.argtypes = [P, i64, P, i32, i64, i32, i32, P, i32, P, P, P]
    lib.pldpo_rank_hidden.argtypes = [P, i32, i64, i64, P, i32, i64, P, P, i32, dbl, P, P, P, P]
    lib.pldpo_rank_attention.argtypes = [P, i32, i32, i64, i64, P, i32, i32, P, i32, i64, P, P, i32,
                                         P, P, P, P]
    lib.pldpo_extract_draft.argtypes = [P, i64, P, i64, P, i32, i32, P, P]
    lib.pldpo_verify_greedy.argtypes = [P, i32, i32, i32, i32, P, P, P, P, P, P, i64, P, i64, P, P]
    lib.pldpo_identify_heads.argtypes = [P, i64, P, i32, i64, i32, P, i32, i32, i64, i64, P, P, P]
    lib.pldpo_rank_hidden_avg.argtypes = [P, i32, i64, i64, i32, P, i32, i64, P, P, i32, ctypes.c_double, P, P,
                                          P, P]
    lib.pldpo_verify_sample.argtypes = [P, i32, i32, i32, i32, ctypes.c_double, P, P, P, P, P, P, P, i64,
                                        P, i64, P, P]
    for f in ("pldpo_find_candidates", "pldpo_rank_hidden", "pldpo_rank_attention",
              "pldpo_extract_draft", "pldpo_verify_greedy", "pldpo_verify_sample", "pldpo_rank_hidden_avg",
              "pldpo_identify_heads"):
        getattr(lib, f).restype = ctypes.c_int


def use_library(path):
    """Point this module at another build of the oracle (e.g. a deliberately
    mutated copy compiled by the pin-strength test).  Returns the previous handle;
    pass ``None`` to go back to the default library."""
    global _lib
    with _lock:
        prev = _lib
        _lib = None
    if path is not None:
        lib = ctypes.CDLL(path)
        _configure(lib)
        with _lock:
            _lib = lib
    return prev


def restore_library(handle):
    global _lib
    with _lock:
        _lib = handle


def _ptr(a):
    # The caller must hold a reference to ``a`` across the foreign call.
    return None if a is None else a.ctypes.data


def _i32(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _elem(a):
    """Return (contiguous array, dtype code).  bf16 is passed as uint16 bit patterns."""
    a = np.ascontiguousarray(a)
    if a.dtype == np.float32:
        return a, F32
    if a.dtype == np.uint16:
        return a, BF16
    raise TypeError(f"oracle takes float32 or bf16-as-uint16 arrays, got {a.dtype}")


def _check(rc, name):
    if rc != 0:
        raise ValueError(f"oracle {name}: invalid arguments (rc={rc})")


def find_candidates(ids, seq_len, ngram_min, ngram_max, C_cap):
    """Eq. 1 + longest-suffix n-gram.  ids: int32 [B, T_cap].  Returns
    (cand_pos [B, C_cap] int32 (unused slots untouched = -1), cand_count [B], match_len [B], status [B])."""
    ids = _i32(ids)
    B, T_cap = ids.shape
    seq_len = _i32(seq_len)
    cand = np.full((B, max(C_cap, 0)), -1, np.int32)
    cnt = np.zeros(B, np.int32)
    ml = np.zeros(B, np.int32)
    st = np.zeros(B, np.uint32)
    _check(_load().pldpo_find_candidates(_ptr(ids), T_cap, _ptr(seq_len), B, T_cap, ngram_min,
                                         ngram_max, _ptr(cand), C_cap, _ptr(cnt), _ptr(ml), _ptr(st)),
           "find_candidates")
    return cand, cnt, ml, st


def rank_hidden(H, seq_len, cand_pos, cand_count, threshold=-np.inf, status=None):
    """Eq. 3.  H: [B, T_cap, d] float32 or bf16 bits (uint16).  Returns
    (scores [B, C_cap] f64, best_pos [B] int32, best_score [B] f64); ``status``
    (numpy uint32 [B]) is OR-ed into when given."""
    H, dt = _elem(H)
    B, T_cap, d = H.shape
    cand_pos = _i32(cand_pos)
    C_cap = cand_pos.shape[1]
    seq_len, cand_count = _i32(seq_len), _i32(cand_count)
    scores = np.full((B, C_cap), np.nan)
    best = np.zeros(B, np.int32)
    bs = np.zeros(B)
    _check(_load().pldpo_rank_hidden(_ptr(H), dt, d, T_cap * d, _ptr(seq_len), B, T_cap, _ptr(cand_pos),
                                     _ptr(cand_count), C_cap, float(threshold), _ptr(scores),
                                     _ptr(best), _ptr(bs), _ptr(status)), "rank_hidden")
    return scores, best, bs


def rank_hidden_avg(H, seq_len, cand_pos, cand_count, m, threshold=-np.inf, status=None):
    """App. B.2: Eq. 3 on window means of the m rows ending at each position.
    Same shapes and returns as rank_hidden."""
    H, dt = _elem(H)
    B, T_cap, d = H.shape
    cand_pos = _i32(cand_pos)
    C_cap = cand_pos.shape[1]
    seq_len, cand_count = _i32(seq_len), _i32(cand_count)
    scores = np.full((B, C_cap), np.nan)
    best = np.zeros(B, np.int32)
    bs = np.zeros(B)
    _check(_load().pldpo_rank_hidden_avg(_ptr(H), dt, d, T_cap * d, int(m), _ptr(seq_len), B, T_cap,
                                         _ptr(cand_pos), _ptr(cand_count), C_cap, float(threshold),
                                         _ptr(scores), _ptr(best), _ptr(bs), _ptr(status)), "rank_hidden_avg")
    return scores, best, bs


def identify_heads(ids, pos, A, max_suffix=64, counts=None):
    """Sec. 4.2.1 head identification.  ids int32 [B, T_cap]; pos int32 [B] (the
    generated token's position p); A [B, R, T_cap] float32 or bf16 bits, the rows of
    query p-1.  Returns (counts uint32 [R] (added to ``counts`` when given), r_star
    int32 [B], status uint32 [B])."""
    ids = _i32(ids)
    B, T_cap = ids.shape
    A, dt = _elem(A)
    R = A.shape[1]
    pos = _i32(pos)
    c = np.zeros(R, np.uint32) if counts is None else counts
    assert c.dtype == np.uint32 and c.flags.c_contiguous and c.size == R
    rs = np.zeros(B, np.int32)
    st = np.zeros(B, np.uint32)
    _check(_load().pldpo_identify_heads(_ptr(ids), T_cap, _ptr(pos), B, T_cap, int(max_suffix), _ptr(A), dt, R,
                                        A.shape[2], R * A.shape[2], _ptr(c), _ptr(rs), _ptr(st)), "identify_heads")
    return c, rs, st


def rank_attention(A, seq_len, cand_pos, cand_count, row_idx=None, agg=AGG_MAX, status=None):
    """Eq. 2.  A: [B, R, T_cap] float32 or bf16 bits (uint16), row r = attention of
    query t-1 for the r-th (layer, head).  Returns (scores, best_pos, best_score)."""
    A, dt = _elem(A)
    B, R, T_cap = A.shape
    cand_pos = _i32(cand_pos)
    C_cap = cand_pos.shape[1]
    ri = None if row_idx is None else _i32(row_idx)
    n_sel = R if ri is None else ri.size
    seq_len, cand_count = _i32(seq_len), _i32(cand_count)
    scores = np.full((B, C_cap), np.nan)
    best = np.zeros(B, np.int32)
    bs = np.zeros(B)
    _check(_load().pldpo_rank_attention(_ptr(A), dt, R, T_cap, R * T_cap, _ptr(ri), n_sel, agg,
                                        _ptr(seq_len), B, T_cap, _ptr(cand_pos), _ptr(cand_count),
                                        C_cap, _ptr(scores), _ptr(best), _ptr(bs), _ptr(status)),
           "rank_attention")
    return scores, best, bs


def extract_draft(ids, seq_len, best_pos, K):
    """Sec. 4.3.  Returns (draft [B, K] int32 padded with -1, draft_len [B])."""
    ids = _i32(ids)
    B, T_cap = ids.shape
    seq_len, best_pos = _i32(seq_len), _i32(best_pos)
    draft = np.zeros((B, K), np.int32)
    dl = np.zeros(B, np.int32)
    _check(_load().pldpo_extract_draft(_ptr(ids), T_cap, _ptr(seq_len), T_cap, _ptr(best_pos), B, K,
                                       _ptr(draft), _ptr(dl)), "extract_draft")
    return draft, dl


def verify_greedy(logits, draft, draft_len, ids=None, seq_len=None, T_cap=None, kv_keep=False):
    """Sec. 4.4, greedy.  logits: [B, K+1, V] float32 or bf16 bits.  ``seq_len``
    (numpy int32, modified IN PLACE) enables the bookkeeping; ``ids`` (numpy int32
    [B, T_cap], modified IN PLACE) the append.  Returns
    dict(argmax, accept_len, next_token, kv_keep_len, status)."""
    logits, dt = _elem(logits)
    B, K1, V = logits.shape
    K = K1 - 1
    draft, draft_len = _i32(draft), _i32(draft_len)
    assert draft.shape == (B, K)
    argmax = np.zeros((B, K1), np.int32)
    acc = np.zeros(B, np.int32)
    nxt = np.zeros(B, np.int32)
    st = np.zeros(B, np.uint32)
    kv = np.zeros(B, np.int32) if kv_keep else None
    stride = 0
    if ids is not None:
        assert ids.dtype == np.int32 and ids.flags.c_contiguous
        T_cap, stride = ids.shape[1], ids.shape[1]
    if seq_len is not None:
        assert seq_len.dtype == np.int32 and seq_len.flags.c_contiguous
        if T_cap is None:
            raise ValueError("seq_len bookkeeping needs T_cap (or ids)")
    _check(_load().pldpo_verify_greedy(_ptr(logits), dt, B, K, V, _ptr(draft), _ptr(draft_len),
                                       _ptr(argmax), _ptr(acc), _ptr(nxt), _ptr(ids), stride,
                                       _ptr(seq_len), int(T_cap or 0), _ptr(kv), _ptr(st)),
           "verify_greedy")
    return dict(argmax=argmax, accept_len=acc, next_token=nxt, kv_keep_len=kv, status=st)


def verify_sample(logits, uniforms, draft, draft_len, temperature=1.0, ids=None, seq_len=None,
                  T_cap=None, kv_keep=False):
    """Sec. 4.4 with sampling at ``temperature``: position i of sequence b draws the
    smallest v whose cumulative softmax(logits / T) probability exceeds
    uniforms[b, i] (float32 [B, K+1]).  Bookkeeping as verify_greedy.  Returns
    dict(sampled, accept_len, next_token, kv_keep_len, status)."""
    logits, dt = _elem(logits)
    B, K1, V = logits.shape
    K = K1 - 1
    draft, draft_len = _i32(draft), _i32(draft_len)
    assert draft.shape == (B, K)
    u = np.ascontiguousarray(uniforms, dtype=np.float32)
    assert u.shape == (B, K1)
    sampled = np.zeros((B, K1), np.int32)
    acc = np.zeros(B, np.int32)
    nxt = np.zeros(B, np.int32)
    st = np.zeros(B, np.uint32)
    kv = np.zeros(B, np.int32) if kv_keep else None
    stride = 0
    if ids is not None:
        assert ids.dtype == np.int32 and ids.flags.c_contiguous
        T_cap, stride = ids.shape[1], ids.shape[1]
    if seq_len is not None:
        assert seq_len.dtype == np.int32 and seq_len.flags.c_contiguous
        if T_cap is None:
            raise ValueError("seq_len bookkeeping needs T_cap (or ids)")
    _check(_load().pldpo_verify_sample(_ptr(logits), dt, B, K, V, float(temperature), _ptr(u), _ptr(draft),
                                       _ptr(draft_len), _ptr(sampled), _ptr(acc), _ptr(nxt), _ptr(ids), stride,
                                       _ptr(seq_len), int(T_cap or 0), _ptr(kv), _ptr(st)),
           "verify_sample")
    return dict(sampled=sampled, accept_len=acc, next_token=nxt, kv_keep_len=kv, status=st)


def bf16_bits(x):
    """fp32 numpy array -> bf16 bit patterns (uint16), round-to-nearest-even.
    Finite inputs only.  Used to hand bf16 data to the oracle."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_to_f32(bits):
    """bf16 bit patterns (uint16) -> exact fp32."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)
