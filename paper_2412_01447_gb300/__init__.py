"""PLD+ drafting and greedy verification on GB300 (sm_103a).

Python binding of the C ABI in ``include/pldp.h``.  Every function here only
marshals torch tensors (device pointers, sizes, the current CUDA stream) into
the library call of the same name; all the work runs in the CUDA kernels of
``libpldp.so``.  There is no CPU fallback: if the library is missing the calls
raise.

PLD+ (arXiv 2412.01447), per decode step and per sequence:
  * ``pldp_find_candidates`` -- Eq. 1 (Sec. 4.2): earlier occurrences of the last
    token, narrowed to the longest matching suffix n-gram;
  * ``pldp_rank_hidden``     -- Eq. 3 (Sec. 4.2.2): cosine of hidden states;
  * ``pldp_rank_attention``  -- Eq. 2 (Sec. 4.2.1): max attention of selected heads;
  * ``pldp_extract_draft``   -- Sec. 4.3: the K tokens after the best occurrence;
  * ``pldp_verify_greedy``   -- Sec. 4.4: greedy accept against the target argmax;
  * ``pldp_verify_sample``   -- Sec. 4.4 with sampling, from caller uniforms.
The fused calls: ``pldp_draft_step`` (the first four in one launch, optionally
with the token index of ``pldp_index_build``), ``pldp_verify_greedy_draft`` and
``pldp_verify_sample_draft`` (verification, greedy or by sampling, then the next
step's draft).  Also ``pldp_rank_hidden_avg``
(App. B.2) and ``pldp_identify_heads`` / ``pldp_top_heads`` (Sec. 4.2.1).

Device buffers are passed as raw pointers, so the binding checks what the C
side cannot: every tensor is a CUDA tensor of the stated dtype, dense where
the call wants it, and holds at least the elements the call will touch.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import _build

__all__ = [
    "build", "library_path", "PldpError",
    "PLDP_F32", "PLDP_BF16", "PLDP_AGG_MAX", "PLDP_AGG_SUM",
    "PLDP_ST_CAND_OVERFLOW", "PLDP_ST_TOKEN_RANGE", "PLDP_ST_CAPACITY", "PLDP_ST_SEQ_LEN",
    "PLDP_ST_DRAFT_LEN", "PLDP_ST_ROW_INDEX", "PLDP_ST_TIMEOUT",
    "PLDP_OK", "PLDP_ERR_INVALID_ARG", "PLDP_ERR_UNSUPPORTED", "PLDP_ERR_CUDA", "PLDP_ERR_TIMEOUT",
    "pldp_find_candidates", "pldp_rank_hidden", "pldp_rank_attention", "pldp_extract_draft",
    "pldp_verify_greedy", "pldp_verify_workspace_size", "pldp_verify_greedy_noalloc",
    "pldp_verify_sample", "pldp_verify_sample_workspace_size",
    "pldp_draft_step", "pldp_draft_step_args", "pldp_draft_workspace_size",
    "pldp_index_size", "pldp_index_build",
    "pldp_verify_greedy_draft", "pldp_verify_draft_args",
    "pldp_verify_sample_draft", "pldp_verify_sample_draft_args", "pldp_verify_sample_draft_workspace_size",
    "pldp_rank_hidden_avg", "pldp_identify_heads", "pldp_top_heads",
    "pldp_version", "pldp_last_error",
]

PLDP_F32, PLDP_BF16 = 0, 1
PLDP_AGG_MAX, PLDP_AGG_SUM = 0, 1
PLDP_ST_CAND_OVERFLOW = 1
PLDP_ST_TOKEN_RANGE = 2
PLDP_ST_CAPACITY = 4
PLDP_ST_SEQ_LEN = 8
PLDP_ST_DRAFT_LEN = 16
PLDP_ST_ROW_INDEX = 32
PLDP_ST_TIMEOUT = 64

PLDP_OK = 0
PLDP_ERR_INVALID_ARG = 1
PLDP_ERR_UNSUPPORTED = 2
PLDP_ERR_CUDA = 3
PLDP_ERR_TIMEOUT = 4

_STATUS_NAMES = {1: "PLDP_ERR_INVALID_ARG", 2: "PLDP_ERR_UNSUPPORTED", 3: "PLDP_ERR_CUDA",
                 4: "PLDP_ERR_TIMEOUT"}


class PldpError(RuntimeError):
    def __init__(self, fn, code, msg):
        super().__init__(f"{fn}: {_STATUS_NAMES.get(code, code)}: {msg}")
        self.code = code


_lock = threading.Lock()
_lib = None


class pldp_draft_step_args(ctypes.Structure):
    """Mirror of the C argument block of pldp_draft_step (include/pldp.h)."""
    _fields_ = [
        ("ids", ctypes.c_void_p), ("ids_stride", ctypes.c_int64), ("seq_len", ctypes.c_void_p),
        ("B", ctypes.c_int), ("T_cap", ctypes.c_int64), ("ngram_min", ctypes.c_int),
        ("ngram_max", ctypes.c_int), ("cand_pos", ctypes.c_void_p), ("C_cap", ctypes.c_int),
        ("cand_count", ctypes.c_void_p), ("match_len", ctypes.c_void_p),
        ("H", ctypes.c_void_p), ("h_dtype", ctypes.c_int), ("d", ctypes.c_int64),
        ("h_seq_stride", ctypes.c_int64), ("threshold", ctypes.c_float), ("h_scores", ctypes.c_void_p),
        ("best_h", ctypes.c_void_p), ("best_h_score", ctypes.c_void_p),
        ("A", ctypes.c_void_p), ("a_dtype", ctypes.c_int), ("R", ctypes.c_int),
        ("a_row_stride", ctypes.c_int64), ("a_key_stride", ctypes.c_int64), ("a_seq_stride", ctypes.c_int64),
        ("row_idx", ctypes.c_void_p),
        ("n_sel", ctypes.c_int), ("agg", ctypes.c_int), ("a_scores", ctypes.c_void_p),
        ("best_a", ctypes.c_void_p), ("best_a_score", ctypes.c_void_p),
        ("draft_from", ctypes.c_int), ("K", ctypes.c_int), ("draft", ctypes.c_void_p),
        ("draft_len", ctypes.c_void_p), ("status", ctypes.c_void_p),
        ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t),
        ("index", ctypes.c_void_p), ("index_bytes", ctypes.c_size_t), ("V", ctypes.c_int),
    ]


class pldp_verify_sample_draft_args(ctypes.Structure):
    """Mirror of the C argument block of pldp_verify_sample_draft (include/pldp.h)."""
    _fields_ = [
        ("logits", ctypes.c_void_p), ("dtype", ctypes.c_int), ("V", ctypes.c_int),
        ("temperature", ctypes.c_float), ("uniforms", ctypes.c_void_p),
        ("draft", ctypes.c_void_p), ("draft_len", ctypes.c_void_p), ("sampled", ctypes.c_void_p),
        ("accept_len", ctypes.c_void_p), ("next_token", ctypes.c_void_p), ("kv_keep_len", ctypes.c_void_p),
        ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t), ("next", pldp_draft_step_args),
    ]


class pldp_verify_draft_args(ctypes.Structure):
    """Mirror of the C argument block of pldp_verify_greedy_draft (include/pldp.h)."""
    _fields_ = [
        ("logits", ctypes.c_void_p), ("dtype", ctypes.c_int), ("V", ctypes.c_int),
        ("draft", ctypes.c_void_p), ("draft_len", ctypes.c_void_p), ("argmax", ctypes.c_void_p),
        ("accept_len", ctypes.c_void_p), ("next_token", ctypes.c_void_p), ("kv_keep_len", ctypes.c_void_p),
        ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t), ("next", pldp_draft_step_args),
    ]


def library_path() -> str:
    return _build.LIB


def build(force: bool = False) -> str:
    """Compile libpldp.so for sm_103a (in-tree) if it is missing or stale."""
    return _build.build(force=force)


def _load():
    global _lib
    if _lib is not None:
        return _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(_build.LIB):
                raise RuntimeError("libpldp.so is not built: call paper_2412_01447_gb300.build() "
                                   "(needs nvcc); there is no CPU fallback")
            lib = ctypes.CDLL(_build.LIB)
            P, i32, i64, f32, sz = (ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float,
                                    ctypes.c_size_t)
            lib.pldp_find_candidates.argtypes = [P, i64, P, i32, i64, i32, i32, P, i32, P, P, P, P]
            lib.pldp_rank_hidden.argtypes = [P, i32, i64, i64, P, i32, i64, P, P, i32, f32, P, P, P,
                                             P, P]
            lib.pldp_identify_heads.argtypes = [P, i64, P, i32, i64, i32, P, i32, i32, i64, i64, P, P, P, P]
            lib.pldp_identify_heads.restype = ctypes.c_int
            lib.pldp_top_heads.argtypes = [P, i32, i32, P, P]
            lib.pldp_top_heads.restype = ctypes.c_int
            lib.pldp_rank_hidden_avg.argtypes = [P, i32, i64, i64, i32, P, i32, i64, P, P, i32, f32, P, P,
                                                 P, P, P]
            lib.pldp_rank_hidden_avg.restype = ctypes.c_int
            lib.pldp_rank_attention.argtypes = [P, i32, i32, i64, i64, i64, P, i32, i32, P, i32, i64, P,
                                                P, i32, P, P, P, P, P]
            lib.pldp_extract_draft.argtypes = [P, i64, P, i64, P, i32, i32, P, P, P]
            lib.pldp_verify_greedy.argtypes = [P, i32, i32, i32, i32, P, P, P, P, P, P, i64, P, i64,
                                               P, P, P, sz, P]
            for f in ("pldp_find_candidates", "pldp_rank_hidden", "pldp_rank_attention",
                      "pldp_extract_draft", "pldp_verify_greedy"):
                getattr(lib, f).restype = ctypes.c_int
            lib.pldp_draft_step.argtypes = [ctypes.POINTER(pldp_draft_step_args), P]
            lib.pldp_draft_step.restype = ctypes.c_int
            lib.pldp_verify_greedy_draft.argtypes = [ctypes.POINTER(pldp_verify_draft_args), P]
            lib.pldp_verify_greedy_draft.restype = ctypes.c_int
            lib.pldp_verify_sample_draft.argtypes = [ctypes.POINTER(pldp_verify_sample_draft_args), P]
            lib.pldp_verify_sample_draft.restype = ctypes.c_int
            lib.pldp_verify_sample_draft_workspace_size.argtypes = [i32, i32, i32, i32]
            lib.pldp_verify_sample_draft_workspace_size.restype = sz
            lib.pldp_draft_workspace_size.argtypes = [i32]
            lib.pldp_draft_workspace_size.restype = sz
            lib.pldp_index_size.argtypes = [i32, i32]
            lib.pldp_index_size.restype = sz
            lib.pldp_index_build.argtypes = [P, i64, P, i32, i64, i32, P, sz, P, P]
            lib.pldp_index_build.restype = ctypes.c_int
            lib.pldp_verify_greedy_noalloc.argtypes = [P, i32, i32, i32, i32, P, P, P, P, P, P, i64,
                                                       P, i64, P, P, P]
            lib.pldp_verify_greedy_noalloc.restype = ctypes.c_int
            lib.pldp_verify_workspace_size.argtypes = [i32, i32, i32]
            lib.pldp_verify_workspace_size.restype = sz
            lib.pldp_verify_sample.argtypes = [P, i32, i32, i32, i32, f32, P, P, P, P, P, P, P, i64, P,
                                               i64, P, P, P, sz, P]
            lib.pldp_verify_sample.restype = ctypes.c_int
            lib.pldp_verify_sample_workspace_size.argtypes = [i32, i32, i32, i32]
            lib.pldp_verify_sample_workspace_size.restype = sz
            lib.pldp_last_error.argtypes = []
            lib.pldp_last_error.restype = ctypes.c_char_p
            lib.pldp_version.argtypes = []
            lib.pldp_version.restype = ctypes.c_int
            _lib = lib
    return _lib


# ----------------------------------------------------------------------------
# marshalling helpers
# ----------------------------------------------------------------------------
def _stream(stream):
    if stream is None:
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, torch.cuda.Stream):
        return ctypes.c_void_p(stream.cuda_stream)
    return ctypes.c_void_p(int(stream))


def _dev(t, name, dtype=None, allow_none=False):
    if t is None:
        if allow_none:
            return None
        raise ValueError(f"{name} is required")
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    return ctypes.c_void_p(t.data_ptr())


_WORD = (torch.int32, getattr(torch, "uint32", torch.int32))


def _dev_or_pinned(t, name):
    """A CUDA tensor, or a page-locked (pinned) host tensor, which the device reads in
    place through unified addressing."""
    if isinstance(t, torch.Tensor) and not t.is_cuda and t.is_pinned():
        return ctypes.c_void_p(t.data_ptr())
    return _dev(t, name)


def _dense(t, name, dtype=None, allow_none=False, n=None):
    """A contiguous tensor of at least n elements (the call reads or writes n).
    dtype _WORD: any 4-byte integer type (status bits, counts)."""
    if t is not None:
        if not isinstance(t, torch.Tensor):
            raise ValueError(f"{name} must be a CUDA tensor")
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")
        if n is not None and t.numel() < n:
            raise ValueError(f"{name} needs {n} elements, has {t.numel()}")
        if dtype is _WORD:
            if t.dtype not in _WORD:
                raise ValueError(f"{name} must be int32 or uint32, got {t.dtype}")
            dtype = None
    return _dev(t, name, dtype, allow_none)


def _rows(t, name, B=None, T_cap=None):
    """A [B, T] int32 tensor whose rows may be strided (unit inner stride), with at
    least B rows; returns (pointer, row stride, T_cap), T_cap at most T (default T)."""
    if not isinstance(t, torch.Tensor) or t.dim() != 2 or t.stride(1) != 1:
        raise ValueError(f"{name} must be 2-D with unit inner stride")
    if B is not None and t.shape[0] < B:
        raise ValueError(f"{name} has {t.shape[0]} rows, the call needs {B}")
    if T_cap is None:
        T_cap = t.shape[1]
    elif not 0 <= T_cap <= t.shape[1]:
        raise ValueError(f"T_cap = {T_cap} is outside [0, {name}.shape[1] = {t.shape[1]}]")
    return _dev(t, name, torch.int32), t.stride(0), int(T_cap)


def _code(x):
    if x in (torch.float32, "f32", PLDP_F32):
        return PLDP_F32
    if x in (torch.bfloat16, "bf16", PLDP_BF16):
        return PLDP_BF16
    raise ValueError(f"unsupported dtype {x}")


def _check(fn, rc):
    if rc != 0:
        raise PldpError(fn, rc, _load().pldp_last_error().decode())


# ----------------------------------------------------------------------------
# the C ABI, one call each
# ----------------------------------------------------------------------------
def pldp_find_candidates(ids, seq_len, ngram_min, ngram_max, cand_pos, cand_count, match_len,
                         status=None, T_cap=None, stream=None):
    """Eq. 1 with the longest-suffix n-gram rule.  ids: int32 [B, T] (rows may be
    strided), seq_len int32 [B]; outputs cand_pos int32 [B, C_cap], cand_count and
    match_len int32 [B], status uint32-as-int32 [B] (optional)."""
    p_ids, stride, T = _rows(ids, "ids", T_cap=T_cap)
    B = ids.shape[0]
    C_cap = cand_pos.shape[1] if cand_pos is not None and cand_pos.dim() == 2 else 0
    _check("pldp_find_candidates", _load().pldp_find_candidates(
        p_ids, stride, _dense(seq_len, "seq_len", torch.int32, n=B), B, T,
        ngram_min, ngram_max, _dense(cand_pos, "cand_pos", torch.int32, allow_none=True, n=B * C_cap), C_cap,
        _dense(cand_count, "cand_count", torch.int32, n=B), _dense(match_len, "match_len", torch.int32, n=B),
        _dense(status, "status", _WORD, allow_none=True, n=B), _stream(stream)))


def pldp_rank_hidden(H, seq_len, cand_pos, cand_count, best_pos, scores=None, best_score=None,
                     threshold=float("-inf"), status=None, stream=None):
    """Eq. 3.  H: [B, T_cap, d] float32/bfloat16 (the chosen layer), contiguous rows;
    cand_pos int32 [B, C_cap]; outputs best_pos int32 [B], scores float32 [B, C_cap]
    and best_score float32 [B] (optional)."""
    if H.dim() != 3 or H.stride(2) != 1 or H.stride(1) != H.shape[2]:
        raise ValueError("H must be [B, T_cap, d] with contiguous rows")
    B, T_cap, d = H.shape
    C_cap = cand_pos.shape[1]
    _check("pldp_rank_hidden", _load().pldp_rank_hidden(
        _dev(H, "H"), _code(H.dtype), d, H.stride(0), _dense(seq_len, "seq_len", torch.int32, n=B), B,
        T_cap, _dense(cand_pos, "cand_pos", torch.int32, n=B * C_cap), _dense(cand_count, "cand_count", torch.int32, n=B),
        C_cap, float(threshold), _dense(scores, "scores", torch.float32, allow_none=True, n=B * C_cap),
        _dense(best_pos, "best_pos", torch.int32, n=B),
        _dense(best_score, "best_score", torch.float32, allow_none=True, n=B),
        _dense(status, "status", _WORD, allow_none=True, n=B), _stream(stream)))


def pldp_rank_hidden_avg(H, seq_len, cand_pos, cand_count, best_pos, m, scores=None, best_score=None,
                         threshold=float("-inf"), status=None, stream=None):
    """App. B.2: Eq. 3 on the means of the m rows ending at each position.  Same
    arguments as pldp_rank_hidden plus the window length m >= 1."""
    if H.dim() != 3 or H.stride(2) != 1 or H.stride(1) != H.shape[2]:
        raise ValueError("H must be [B, T_cap, d] with contiguous rows")
    B, T_cap, d = H.shape
    C_cap = cand_pos.shape[1]
    _check("pldp_rank_hidden_avg", _load().pldp_rank_hidden_avg(
        _dev(H, "H"), _code(H.dtype), d, H.stride(0), int(m), _dense(seq_len, "seq_len", torch.int32, n=B), B,
        T_cap, _dense(cand_pos, "cand_pos", torch.int32, n=B * C_cap), _dense(cand_count, "cand_count", torch.int32, n=B),
        C_cap, float(threshold), _dense(scores, "scores", torch.float32, allow_none=True, n=B * C_cap),
        _dense(best_pos, "best_pos", torch.int32, n=B),
        _dense(best_score, "best_score", torch.float32, allow_none=True, n=B),
        _dense(status, "status", _WORD, allow_none=True, n=B), _stream(stream)))


def pldp_identify_heads(ids, pos, A, counts, max_suffix=64, r_star=None, status=None, stream=None):
    """Sec. 4.2.1 head identification.  ids int32 [B, T_cap]; pos int32 [B] (the
    generated token's position p); A [B, R, T_cap] float32/bfloat16, the attention
    rows of query p-1 (unit inner stride); counts int32/uint32 [R] CUDA tensor,
    added to.  r_star int32 [B] out (optional)."""
    if A.dim() != 3 or A.stride(2) != 1:
        raise ValueError("A must be [B, R, T_cap] with unit inner stride")
    B, R = A.shape[0], A.shape[1]
    p_ids, stride, T_cap = _rows(ids, "ids", B)
    if A.shape[2] < T_cap:
        raise ValueError("A must cover the T_cap = ids.shape[1] key positions")
    _check("pldp_identify_heads", _load().pldp_identify_heads(
        p_ids, stride, _dense(pos, "pos", torch.int32, n=B), B, T_cap, int(max_suffix), _dev(A, "A"), _code(A.dtype),
        R, A.stride(1), A.stride(0), _dense(counts, "counts", _WORD, n=R),
        _dense(r_star, "r_star", torch.int32, allow_none=True, n=B),
        _dense(status, "status", _WORD, allow_none=True, n=B), _stream(stream)))


def pldp_top_heads(counts, k, row_idx, stream=None):
    """The k rows with the most counts (ties to the smaller index) into row_idx int32 [k]."""
    _check("pldp_top_heads", _load().pldp_top_heads(_dense(counts, "counts", _WORD), counts.numel(), int(k),
                                                    _dense(row_idx, "row_idx", torch.int32, n=int(k)),
                                                    _stream(stream)))


def pldp_rank_attention(A, seq_len, cand_pos, cand_count, best_pos, row_idx=None, agg=PLDP_AGG_MAX,
                        scores=None, best_score=None, status=None, stream=None):
    """Eq. 2.  A: [B, R, T_cap] float32/bfloat16, attention of query t-1 for each of R
    (layer, head) rows, with contiguous keys (each row dense) or key-major (the R values
    of a key dense: e.g. a [B, T_cap, R] tensor transposed to [B, R, T_cap]), on the
    device or in pinned host memory (read in place: only the selected rows' values at the
    candidate keys cross the link); row_idx int32 [n_sel] device or None (all)."""
    if A.dim() != 3:
        raise ValueError("A must be [B, R, T_cap]")
    B, R, T_cap = A.shape
    C_cap = cand_pos.shape[1]
    n_sel = R if row_idx is None else row_idx.numel()
    _check("pldp_rank_attention", _load().pldp_rank_attention(
        _dev_or_pinned(A, "A"), _code(A.dtype), R, A.stride(1), A.stride(2), A.stride(0),
        _dense(row_idx, "row_idx", torch.int32, allow_none=True), n_sel, int(agg),
        _dense(seq_len, "seq_len", torch.int32, n=B), B, T_cap, _dense(cand_pos, "cand_pos", torch.int32, n=B * C_cap),
        _dense(cand_count, "cand_count", torch.int32, n=B), C_cap,
        _dense(scores, "scores", torch.float32, allow_none=True, n=B * C_cap),
        _dense(best_pos, "best_pos", torch.int32, n=B),
        _dense(best_score, "best_score", torch.float32, allow_none=True, n=B),
        _dense(status, "status", _WORD, allow_none=True, n=B), _stream(stream)))


def pldp_extract_draft(ids, seq_len, best_pos, draft, draft_len, T_cap=None, stream=None):
    """Sec. 4.3.  draft int32 [B, K] and draft_len int32 [B] are written."""
    B, K = draft.shape
    p_ids, stride, T = _rows(ids, "ids", B, T_cap)
    _check("pldp_extract_draft", _load().pldp_extract_draft(
        p_ids, stride, _dense(seq_len, "seq_len", torch.int32, n=B), T,
        _dense(best_pos, "best_pos", torch.int32, n=B), B, K, _dense(draft, "draft", torch.int32, n=B * K),
        _dense(draft_len, "draft_len", torch.int32, n=B), _stream(stream)))


def pldp_draft_workspace_size(B) -> int:
    return int(_load().pldp_draft_workspace_size(B))


def _draft_args(ids, seq_len, ngram_min, ngram_max, cand_pos, cand_count, match_len, K, draft,
                draft_len, workspace, H=None, best_h=None, h_scores=None, best_h_score=None,
                threshold=float("-inf"), A=None, best_a=None, row_idx=None, agg=PLDP_AGG_MAX,
                a_scores=None, best_a_score=None, draft_from="hidden", status=None, T_cap=None,
                index=None, V=None):
    """The argument block of pldp_draft_step (marshalling only)."""
    p_ids, stride, T = _rows(ids, "ids", T_cap=T_cap)
    B = ids.shape[0]
    a = pldp_draft_step_args()
    a.ids, a.ids_stride, a.seq_len, a.B = p_ids, stride, _dense(seq_len, "seq_len", torch.int32, n=B), B
    a.T_cap = T
    a.ngram_min, a.ngram_max = ngram_min, ngram_max
    a.C_cap = C_cap = cand_pos.shape[1] if cand_pos is not None and cand_pos.dim() == 2 else 0
    a.cand_pos = _dense(cand_pos, "cand_pos", torch.int32, allow_none=True, n=B * C_cap)
    a.cand_count = _dense(cand_count, "cand_count", torch.int32, n=B)
    a.match_len = _dense(match_len, "match_len", torch.int32, n=B)
    if H is not None:
        if H.dim() != 3 or H.stride(2) != 1 or H.stride(1) != H.shape[2]:
            raise ValueError("H must be [B, T_cap, d] with contiguous rows")
        if H.shape[0] < B or H.shape[1] < T:
            raise ValueError(f"H must cover [B, T_cap] = [{B}, {T}] positions")
        a.H, a.h_dtype, a.d, a.h_seq_stride = _dev(H, "H"), _code(H.dtype), H.shape[2], H.stride(0)
        a.threshold = float(threshold)
        a.h_scores = _dense(h_scores, "h_scores", torch.float32, allow_none=True, n=B * C_cap)
        a.best_h = _dense(best_h, "best_h", torch.int32, n=B)
        a.best_h_score = _dense(best_h_score, "best_h_score", torch.float32, allow_none=True, n=B)
    if A is not None:
        if A.dim() != 3:
            raise ValueError("A must be [B, R, T_cap]")
        if A.shape[0] < B or A.shape[2] < T:
            raise ValueError(f"A must cover [B, T_cap] = [{B}, {T}] positions")
        a.A, a.a_dtype, a.R = _dev_or_pinned(A, "A"), _code(A.dtype), A.shape[1]
        a.a_row_stride, a.a_key_stride, a.a_seq_stride = A.stride(1), A.stride(2), A.stride(0)
        a.row_idx = _dense(row_idx, "row_idx", torch.int32, allow_none=True)
        a.n_sel = A.shape[1] if row_idx is None else row_idx.numel()
        a.agg = int(agg)
        a.a_scores = _dense(a_scores, "a_scores", torch.float32, allow_none=True, n=B * C_cap)
        a.best_a = _dense(best_a, "best_a", torch.int32, n=B)
        a.best_a_score = _dense(best_a_score, "best_a_score", torch.float32, allow_none=True, n=B)
    a.draft_from = {"hidden": 0, "attention": 1, 0: 0, 1: 1}[draft_from]
    a.K = K
    a.draft = _dense(draft, "draft", torch.int32, n=B * K)
    a.draft_len = _dense(draft_len, "draft_len", torch.int32, n=B)
    a.status = _dense(status, "status", _WORD, allow_none=True, n=B)
    if workspace is not None:
        a.workspace = _dense(workspace, "workspace")
        a.workspace_bytes = workspace.numel() * workspace.element_size()
    if index is not None:
        if V is None:
            raise ValueError("an index needs V")
        a.index = _dense(index, "index")
        a.index_bytes = index.numel() * index.element_size()
        a.V = int(V)
    return a


def pldp_draft_step(ids, seq_len, ngram_min, ngram_max, cand_pos, cand_count, match_len, K, draft,
                    draft_len, workspace, stream=None, **kw):
    """Candidate search, ranking (hidden and/or attention) and draft in one call; the
    arguments mean what they mean in the separate calls.  workspace: a uint8 CUDA
    tensor of pldp_draft_workspace_size(B) bytes, zeroed once before first use (may be
    None with an index).  index: a uint8 CUDA tensor of pldp_index_size(B, V) bytes
    built by pldp_index_build (token ids in [0, V)); the step then looks occurrences
    up instead of scanning, with the same results.  Keyword arguments: H, best_h,
    h_scores, best_h_score, threshold, A, best_a, row_idx, agg, a_scores,
    best_a_score, draft_from, status, T_cap, index, V."""
    a = _draft_args(ids, seq_len, ngram_min, ngram_max, cand_pos, cand_count, match_len, K, draft,
                    draft_len, workspace, **kw)
    _check("pldp_draft_step", _load().pldp_draft_step(ctypes.byref(a), _stream(stream)))


def pldp_verify_greedy_draft(logits, draft, draft_len, accept_len, next_token, workspace, ids, seq_len,
                             ngram_min, ngram_max, cand_pos, cand_count, match_len, next_draft,
                             next_draft_len, index, argmax=None, kv_keep_len=None, stream=None, **kw):
    """Greedy verification of this step (as pldp_verify_greedy, appending to ids and
    seq_len) followed by the next step's drafting with the token index (as
    pldp_draft_step on the extended context), in one call.  next_draft /
    next_draft_len receive the next draft (they may be draft / draft_len).  Keyword
    arguments are pldp_draft_step's (H, best_h, A, best_a, status, ...)."""
    B, K1, V = logits.shape
    K = K1 - 1
    if draft.shape != (B, K) or next_draft.shape != (B, K):
        raise ValueError("draft and next_draft must be [B, K] with K = logits.shape[1] - 1")
    if not isinstance(ids, torch.Tensor) or ids.dim() != 2 or ids.shape[0] != B:
        raise ValueError("ids must be [B, T_cap] with B = logits.shape[0]")
    a = pldp_verify_draft_args()
    a.next = _draft_args(ids, seq_len, ngram_min, ngram_max, cand_pos, cand_count, match_len, K, next_draft,
                         next_draft_len, None, index=index, V=V, **kw)
    a.logits, a.dtype, a.V = _dense(logits, "logits"), _code(logits.dtype), V
    a.draft = _dense(draft, "draft", torch.int32, n=B * K)
    a.draft_len = _dense(draft_len, "draft_len", torch.int32, n=B)
    a.argmax = _dense(argmax, "argmax", torch.int32, allow_none=True, n=B * K1)
    a.accept_len = _dense(accept_len, "accept_len", torch.int32, n=B)
    a.next_token = _dense(next_token, "next_token", torch.int32, n=B)
    a.kv_keep_len = _dense(kv_keep_len, "kv_keep_len", torch.int32, allow_none=True, n=B)
    a.workspace = _dense(workspace, "workspace")
    a.workspace_bytes = workspace.numel() * workspace.element_size()
    _check("pldp_verify_greedy_draft", _load().pldp_verify_greedy_draft(ctypes.byref(a), _stream(stream)))


def pldp_verify_sample_draft_workspace_size(B, K, V, dtype=torch.bfloat16) -> int:
    return int(_load().pldp_verify_sample_draft_workspace_size(B, K, V, _code(dtype)))


def pldp_verify_sample_draft(logits, uniforms, draft, draft_len, accept_len, next_token, workspace, ids, seq_len,
                             ngram_min, ngram_max, cand_pos, cand_count, match_len, next_draft, next_draft_len,
                             index, temperature=1.0, sampled=None, kv_keep_len=None, stream=None, **kw):
    """Sampling verification of this step (as pldp_verify_sample at ``temperature``
    with ``uniforms`` [B, K+1], appending to ids and seq_len) followed by the next
    step's drafting with the token index (as pldp_draft_step on the extended
    context), in one call.  workspace: uint8 CUDA tensor of
    pldp_verify_sample_draft_workspace_size(B, K, V, dtype) bytes.  Other arguments
    as pldp_verify_greedy_draft."""
    B, K1, V = logits.shape
    K = K1 - 1
    if draft.shape != (B, K) or next_draft.shape != (B, K):
        raise ValueError("draft and next_draft must be [B, K] with K = logits.shape[1] - 1")
    if uniforms.shape != (B, K1):
        raise ValueError("uniforms must be [B, K+1]")
    if not isinstance(ids, torch.Tensor) or ids.dim() != 2 or ids.shape[0] != B:
        raise ValueError("ids must be [B, T_cap] with B = logits.shape[0]")
    a = pldp_verify_sample_draft_args()
    a.next = _draft_args(ids, seq_len, ngram_min, ngram_max, cand_pos, cand_count, match_len, K, next_draft,
                         next_draft_len, None, index=index, V=V, **kw)
    a.logits, a.dtype, a.V = _dense(logits, "logits"), _code(logits.dtype), V
    a.temperature = float(temperature)
    a.uniforms = _dense(uniforms, "uniforms", torch.float32, n=B * K1)
    a.draft = _dense(draft, "draft", torch.int32, n=B * K)
    a.draft_len = _dense(draft_len, "draft_len", torch.int32, n=B)
    a.sampled = _dense(sampled, "sampled", torch.int32, allow_none=True, n=B * K1)
    a.accept_len = _dense(accept_len, "accept_len", torch.int32, n=B)
    a.next_token = _dense(next_token, "next_token", torch.int32, n=B)
    a.kv_keep_len = _dense(kv_keep_len, "kv_keep_len", torch.int32, allow_none=True, n=B)
    a.workspace = _dense(workspace, "workspace")
    a.workspace_bytes = workspace.numel() * workspace.element_size()
    _check("pldp_verify_sample_draft", _load().pldp_verify_sample_draft(ctypes.byref(a), _stream(stream)))


def pldp_index_size(B, V) -> int:
    return int(_load().pldp_index_size(B, V))


def pldp_index_build(ids, seq_len, V, index, status=None, T_cap=None, stream=None):
    """Builds the incremental token index of pldp_draft_step over positions
    0 .. seq_len[b]-2 of every sequence.  index: uint8 CUDA tensor of
    pldp_index_size(B, V) bytes (cleared by the call)."""
    p_ids, stride, T = _rows(ids, "ids", T_cap=T_cap)
    B = ids.shape[0]
    _check("pldp_index_build", _load().pldp_index_build(
        p_ids, stride, _dense(seq_len, "seq_len", torch.int32, n=B), B, T, int(V),
        _dense(index, "index"), index.numel() * index.element_size(),
        _dense(status, "status", _WORD, allow_none=True, n=B), _stream(stream)))


def pldp_verify_workspace_size(B, K, V) -> int:
    return int(_load().pldp_verify_workspace_size(B, K, V))


def pldp_verify_greedy(logits, draft, draft_len, accept_len, next_token, workspace, argmax=None,
                       ids=None, seq_len=None, kv_keep_len=None, status=None, T_cap=None,
                       stream=None):
    """Sec. 4.4 (greedy).  logits [B, K+1, V] float32/bfloat16 contiguous; workspace a
    uint8 CUDA tensor of pldp_verify_workspace_size(B, K, V) bytes, zeroed once before
    first use (every call leaves it zeroed).  ids/seq_len (optional, modified in place)
    get the accepted tokens and the bonus token appended."""
    B, K1, V = logits.shape
    K = K1 - 1
    if draft.shape != (B, K):
        raise ValueError("draft must be [B, K] with K = logits.shape[1] - 1")
    p_ids, stride, T = (None, 0, 0) if ids is None else _rows(ids, "ids", B, T_cap)
    if T_cap is None:
        T_cap = T
    _check("pldp_verify_greedy", _load().pldp_verify_greedy(
        _dense(logits, "logits"), _code(logits.dtype), B, K, V, _dense(draft, "draft", torch.int32, n=B * K),
        _dense(draft_len, "draft_len", torch.int32, n=B),
        _dense(argmax, "argmax", torch.int32, allow_none=True, n=B * K1),
        _dense(accept_len, "accept_len", torch.int32, n=B), _dense(next_token, "next_token", torch.int32, n=B),
        p_ids, stride, _dense(seq_len, "seq_len", torch.int32, allow_none=True, n=B), T_cap,
        _dense(kv_keep_len, "kv_keep_len", torch.int32, allow_none=True, n=B),
        _dense(status, "status", _WORD, allow_none=True, n=B), _dense(workspace, "workspace"),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def pldp_verify_sample_workspace_size(B, K, V, dtype=torch.bfloat16) -> int:
    return int(_load().pldp_verify_sample_workspace_size(B, K, V, _code(dtype)))


def pldp_verify_sample(logits, uniforms, draft, draft_len, accept_len, next_token, workspace,
                       temperature=1.0, sampled=None, ids=None, seq_len=None, kv_keep_len=None,
                       status=None, T_cap=None, stream=None):
    """Sec. 4.4 with sampling at ``temperature``: position i of sequence b draws the
    smallest v whose cumulative softmax(logits / T) probability exceeds uniforms[b, i]
    (float32 [B, K+1] CUDA tensor); acceptance and bookkeeping as pldp_verify_greedy.
    workspace: uint8 CUDA tensor of pldp_verify_sample_workspace_size(B, K, V, dtype) bytes."""
    B, K1, V = logits.shape
    K = K1 - 1
    if draft.shape != (B, K):
        raise ValueError("draft must be [B, K] with K = logits.shape[1] - 1")
    if uniforms.shape != (B, K1):
        raise ValueError("uniforms must be [B, K+1]")
    p_ids, stride, T = (None, 0, 0) if ids is None else _rows(ids, "ids", B, T_cap)
    if T_cap is None:
        T_cap = T
    _check("pldp_verify_sample", _load().pldp_verify_sample(
        _dense(logits, "logits"), _code(logits.dtype), B, K, V, float(temperature),
        _dense(uniforms, "uniforms", torch.float32), _dense(draft, "draft", torch.int32, n=B * K),
        _dense(draft_len, "draft_len", torch.int32, n=B), _dense(sampled, "sampled", torch.int32, allow_none=True, n=B * K1),
        _dense(accept_len, "accept_len", torch.int32, n=B), _dense(next_token, "next_token", torch.int32, n=B),
        p_ids, stride, _dense(seq_len, "seq_len", torch.int32, allow_none=True, n=B), T_cap,
        _dense(kv_keep_len, "kv_keep_len", torch.int32, allow_none=True, n=B),
        _dense(status, "status", _WORD, allow_none=True, n=B), _dense(workspace, "workspace"),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def pldp_verify_greedy_noalloc(logits, draft, draft_len, accept_len, next_token, argmax=None,
                               ids=None, seq_len=None, kv_keep_len=None, status=None, T_cap=None,
                               stream=None):
    """pldp_verify_greedy for callers that cannot allocate a workspace: the library
    uses its own fixed scratch area (see include/pldp.h for the size limit and for
    why overlapping calls on one device must be serialised)."""
    B, K1, V = logits.shape
    K = K1 - 1
    if draft.shape != (B, K):
        raise ValueError("draft must be [B, K] with K = logits.shape[1] - 1")
    p_ids, stride, T = (None, 0, 0) if ids is None else _rows(ids, "ids", B, T_cap)
    if T_cap is None:
        T_cap = T
    _check("pldp_verify_greedy_noalloc", _load().pldp_verify_greedy_noalloc(
        _dense(logits, "logits"), _code(logits.dtype), B, K, V, _dense(draft, "draft", torch.int32, n=B * K),
        _dense(draft_len, "draft_len", torch.int32, n=B),
        _dense(argmax, "argmax", torch.int32, allow_none=True, n=B * K1),
        _dense(accept_len, "accept_len", torch.int32, n=B), _dense(next_token, "next_token", torch.int32, n=B),
        p_ids, stride, _dense(seq_len, "seq_len", torch.int32, allow_none=True, n=B), T_cap,
        _dense(kv_keep_len, "kv_keep_len", torch.int32, allow_none=True, n=B),
        _dense(status, "status", _WORD, allow_none=True, n=B), _stream(stream)))


def pldp_version() -> int:
    return int(_load().pldp_version())


def pldp_last_error() -> str:
    return _load().pldp_last_error().decode()
