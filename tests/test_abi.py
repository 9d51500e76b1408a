"""The C ABI library loads without a GPU and exports every call include/pldp.h
declares; host-side argument checks fail before anything touches CUDA."""
import ctypes
import os
import re

import pytest

import paper_2412_01447_gb300 as pk

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "pldp.h")


def declared_symbols():
    src = open(HEADER).read()
    return sorted(set(re.findall(r"PLDP_API\s+[\w\s\*]+?\b(pldp_\w+)\s*\(", src)))


@pytest.fixture(scope="module")
def so():
    pk.build()
    return ctypes.CDLL(pk.library_path())


def test_header_declares_the_five_steps():
    names = declared_symbols()
    for n in ("pldp_find_candidates", "pldp_rank_hidden", "pldp_rank_attention",
              "pldp_extract_draft", "pldp_verify_greedy"):
        assert n in names


def test_exports_every_declared_symbol(so):
    for name in declared_symbols():
        assert hasattr(so, name), name


def test_no_stray_exports(so):
    out = os.popen(f"nm -D --defined-only {pk.library_path()}").read()
    exported = sorted(set(re.findall(r"\b(pldp_\w+)\b", out)))
    assert exported == declared_symbols()


def test_version_and_workspace_are_host_only():
    assert pk.pldp_version() == 200
    assert pk.pldp_verify_workspace_size(0, 1, 1) == 0 + 0
    n = pk.pldp_verify_workspace_size(128, 12, 128256)
    assert n >= 128 * 13 * 8 and n % 256 == 0                  # one 64-bit key per logits row
    assert pk.pldp_verify_workspace_size(4, 0, 10) == 0


def test_host_argument_checks(so):
    lib = pk._load()
    null = None
    # find_candidates: B < 0, bad n-gram range, stride < T_cap
    assert lib.pldp_find_candidates(null, 8, null, -1, 8, 1, 3, null, 4, null, null, null, null) == 1
    assert lib.pldp_find_candidates(null, 8, null, 1, 8, 2, 1, null, 4, null, null, null, null) == 1
    assert lib.pldp_find_candidates(null, 8, null, 1, 8, 1, 9, null, 4, null, null, null, null) == 1
    assert lib.pldp_find_candidates(null, 4, null, 1, 8, 1, 3, null, 4, null, null, null, null) == 1
    assert "ids_stride" in pk.pldp_last_error()
    assert lib.pldp_find_candidates(null, 8, null, 1, 8, 1, 3, null, 4, null, null, null, null) == 1
    assert "null" in pk.pldp_last_error()
    assert lib.pldp_find_candidates(null, 8, null, 0, 8, 1, 3, null, 4, null, null, null, null) == 0
    # rank_hidden: unsupported dtype, d too large, NaN threshold
    args = [null, 0, 64, 64 * 8, null, 1, 8, null, null, 4, float("-inf"), null, null, null, null, null]
    bad = list(args); bad[1] = 7
    assert lib.pldp_rank_hidden(*bad) == 2
    bad = list(args); bad[2] = 1 << 20; bad[3] = (1 << 20) * 8
    assert lib.pldp_rank_hidden(*bad) == 2
    bad = list(args); bad[10] = float("nan")
    assert lib.pldp_rank_hidden(*bad) == 1
    # rank_hidden_avg: m < 1, d too large for the fp32 query sum
    av = [null, 1, 64, 64 * 8, 2, null, 1, 8, null, null, 4, float("-inf"), null, null, null, null, null]
    bad = list(av); bad[4] = 0
    assert lib.pldp_rank_hidden_avg(*bad) == 1 and "m < 1" in pk.pldp_last_error()
    bad = list(av); bad[2] = 49153; bad[3] = 49153 * 8
    assert lib.pldp_rank_hidden_avg(*bad) == 2
    # identify_heads: max_suffix < 1, row_stride < T_cap; top_heads: k > R
    ih = [null, 16, null, 2, 16, 8, null, 1, 4, 16, 64, null, null, null, null]
    bad = list(ih); bad[5] = 0
    assert lib.pldp_identify_heads(*bad) == 1 and "max_suffix" in pk.pldp_last_error()
    bad = list(ih); bad[9] = 8
    assert lib.pldp_identify_heads(*bad) == 1 and "row_stride" in pk.pldp_last_error()
    assert lib.pldp_top_heads(ctypes.c_void_p(256), 4, 5, ctypes.c_void_p(256), null) == 1
    assert lib.pldp_top_heads(ctypes.c_void_p(256), 9000, 5, ctypes.c_void_p(256), null) == 1
    # rank_attention: bad aggregation, n_sel out of range, overlapping or short layouts
    a = [null, 1, 4, 8, 1, 32, null, 4, 0, null, 1, 8, null, null, 4, null, null, null, null, null]
    bad = list(a); bad[8] = 5
    assert lib.pldp_rank_attention(*bad) == 1
    bad = list(a); bad[6] = ctypes.c_void_p(16); bad[7] = 0
    assert lib.pldp_rank_attention(*bad) == 1
    bad = list(a); bad[3], bad[4] = 2, 2                  # rows of 8 keys 2 apart, 2 apart: they overlap
    assert lib.pldp_rank_attention(*bad) == 1 and "overlap" in pk.pldp_last_error()
    bad = list(a); bad[5] = 31                            # one element short of the 4 rows of 8 keys
    assert lib.pldp_rank_attention(*bad) == 1 and "seq_stride" in pk.pldp_last_error()
    ok = list(a); ok[3], ok[4], ok[5] = 1, 4, 32          # key-major: the 4 values of a key side by side
    assert lib.pldp_rank_attention(*ok) == 1 and "null" in pk.pldp_last_error()   # layout passes; no buffers
    # extract_draft: K < 1
    assert lib.pldp_extract_draft(null, 8, null, 8, null, 1, 0, null, null, null) == 1
    # verify_greedy: K < 1, ids without seq_len, workspace too small
    v = [null, 1, 2, 4, 100, null, null, null, null, null, null, 0, null, 0, null, null, null, 0, null]
    bad = list(v); bad[3] = 0
    assert lib.pldp_verify_greedy(*bad) == 1
    bad = list(v); bad[10] = ctypes.c_void_p(16)
    assert lib.pldp_verify_greedy(*bad) == 1
    bad = list(v)
    for k in (0, 5, 6, 8, 9):
        bad[k] = ctypes.c_void_p(256)
    bad[16] = ctypes.c_void_p(256); bad[17] = 8
    assert lib.pldp_verify_greedy(*bad) == 1
    assert "workspace" in pk.pldp_last_error()
    # verify_sample: temperature not positive/finite, K < 1, workspace too small
    sm = [null, 1, 2, 4, 100, 1.0, null, null, null, null, null, null, null, 0, null, 0, null, null, null, 0,
          null]
    for t in (0.0, -1.0, float("inf"), float("nan")):
        bad = list(sm); bad[5] = t
        assert lib.pldp_verify_sample(*bad) == 1 and "temperature" in pk.pldp_last_error()
    bad = list(sm); bad[3] = 0
    assert lib.pldp_verify_sample(*bad) == 1
    bad = list(sm)
    for k in (0, 6, 7, 8, 10, 11):
        bad[k] = ctypes.c_void_p(256)
    bad[18] = ctypes.c_void_p(256); bad[19] = 8
    assert lib.pldp_verify_sample(*bad) == 1 and "workspace" in pk.pldp_last_error()
    assert lib.pldp_verify_sample_workspace_size(2, 4, 100, 7) == 0
    assert lib.pldp_verify_sample_workspace_size(128, 12, 128256, 1) == 128 * 13 * 126 * 8


def test_python_binding_refuses_cpu_tensors():
    import torch
    x = torch.zeros((2, 8), dtype=torch.int32)
    with pytest.raises(ValueError):
        pk.pldp_find_candidates(x, torch.zeros(2, dtype=torch.int32), 1, 3,
                                torch.zeros((2, 4), dtype=torch.int32),
                                torch.zeros(2, dtype=torch.int32), torch.zeros(2, dtype=torch.int32))


def test_draft_step_args_layout_matches_header(tmp_path):
    """The Python mirror of pldp_draft_step_args has the C layout (gcc offsetof)."""
    names = [f for f, _ in pk.pldp_draft_step_args._fields_]
    src = ['#include <stdio.h>', '#include <stddef.h>', f'#include "{HEADER}"', "int main(void) {",
           'printf("%zu\\n", sizeof(pldp_draft_step_args));']
    src += [f'printf("%zu\\n", offsetof(pldp_draft_step_args, {n}));' for n in names]
    src += ["return 0; }"]
    c = tmp_path / "layout.c"
    c.write_text("\n".join(src))
    exe = tmp_path / "layout"
    import subprocess
    subprocess.check_call(["gcc", str(c), "-o", str(exe)])
    out = [int(x) for x in subprocess.check_output([str(exe)]).split()]
    assert out[0] == ctypes.sizeof(pk.pldp_draft_step_args)
    for n, off in zip(names, out[1:]):
        assert getattr(pk.pldp_draft_step_args, n).offset == off, n


@pytest.mark.parametrize("struct", ["pldp_verify_draft_args", "pldp_verify_sample_draft_args"])
def test_verify_draft_args_layout_matches_header(tmp_path, struct):
    """The Python mirrors of the fused verification + next draft argument blocks (with
    their nested draft block) have the C layout (gcc offsetof)."""
    cls = getattr(pk, struct)
    names = [f for f, _ in cls._fields_]
    src = ['#include <stdio.h>', '#include <stddef.h>', f'#include "{HEADER}"', "int main(void) {",
           f'printf("%zu\\n", sizeof({struct}));']
    src += [f'printf("%zu\\n", offsetof({struct}, {n}));' for n in names]
    src += ["return 0; }"]
    c = tmp_path / "layout2.c"
    c.write_text("\n".join(src))
    exe = tmp_path / "layout2"
    import subprocess
    subprocess.check_call(["gcc", str(c), "-o", str(exe)])
    out = [int(x) for x in subprocess.check_output([str(exe)]).split()]
    assert out[0] == ctypes.sizeof(cls)
    for n, off in zip(names, out[1:]):
        assert getattr(cls, n).offset == off, n


def test_verify_draft_host_checks(so):
    """pldp_verify_greedy_draft refuses, before any launch: a null block, a missing
    index, an index sized for another vocabulary, a bad dtype, the draft step's own
    argument errors, missing verification buffers and a short workspace; B == 0 is a
    no-op."""
    lib = pk._load()
    P = ctypes.c_void_p

    def block():
        a = pk.pldp_verify_draft_args()
        n = a.next
        n.ids, n.ids_stride, n.seq_len, n.B, n.T_cap = P(256), 64, P(256), 2, 64
        n.ngram_min, n.ngram_max, n.cand_pos, n.C_cap = 1, 3, P(256), 8
        n.cand_count, n.match_len = P(256), P(256)
        n.H, n.h_dtype, n.d, n.h_seq_stride, n.threshold, n.best_h = P(256), 1, 64, 64 * 64, float("-inf"), P(256)
        n.draft_from, n.K, n.draft, n.draft_len = 0, 4, P(256), P(256)
        n.index, n.index_bytes, n.V = P(256), pk.pldp_index_size(2, 100), 100
        a.logits, a.dtype, a.V = P(256), 1, 100
        a.draft, a.draft_len, a.accept_len, a.next_token = P(256), P(256), P(256), P(256)
        a.workspace, a.workspace_bytes = P(256), pk.pldp_verify_workspace_size(2, 4, 100)
        return a

    def call(a):
        return lib.pldp_verify_greedy_draft(ctypes.byref(a), None)

    assert lib.pldp_verify_greedy_draft(None, None) == pk.PLDP_ERR_INVALID_ARG
    a = block(); a.next.index = None
    assert call(a) == pk.PLDP_ERR_INVALID_ARG and "index" in pk.pldp_last_error()
    a = block(); a.next.V = 99
    assert call(a) == pk.PLDP_ERR_INVALID_ARG and "V" in pk.pldp_last_error()
    a = block(); a.dtype = 7
    assert call(a) == pk.PLDP_ERR_UNSUPPORTED
    a = block(); a.next.ngram_max = 0
    assert call(a) == pk.PLDP_ERR_INVALID_ARG and "verify_greedy_draft" in pk.pldp_last_error()
    a = block(); a.next.index_bytes = 64
    assert call(a) == pk.PLDP_ERR_INVALID_ARG and "index needs" in pk.pldp_last_error()
    a = block(); a.accept_len = None
    assert call(a) == pk.PLDP_ERR_INVALID_ARG and "null" in pk.pldp_last_error()
    a = block(); a.workspace_bytes = 8
    assert call(a) == pk.PLDP_ERR_INVALID_ARG and "workspace" in pk.pldp_last_error()
    a = block(); a.next.B = 0
    assert call(a) == pk.PLDP_OK


def test_verify_sample_draft_host_checks(so):
    """pldp_verify_sample_draft refuses, before any launch: a null block, a missing
    index, a bad temperature, missing uniforms, the draft step's own argument errors
    and a short workspace; B == 0 is a no-op."""
    lib = pk._load()
    P = ctypes.c_void_p

    def block():
        a = pk.pldp_verify_sample_draft_args()
        n = a.next
        n.ids, n.ids_stride, n.seq_len, n.B, n.T_cap = P(256), 64, P(256), 2, 64
        n.ngram_min, n.ngram_max, n.cand_pos, n.C_cap = 1, 3, P(256), 8
        n.cand_count, n.match_len = P(256), P(256)
        n.H, n.h_dtype, n.d, n.h_seq_stride, n.threshold, n.best_h = P(256), 1, 64, 64 * 64, float("-inf"), P(256)
        n.draft_from, n.K, n.draft, n.draft_len = 0, 4, P(256), P(256)
        n.index, n.index_bytes, n.V = P(256), pk.pldp_index_size(2, 100), 100
        a.logits, a.dtype, a.V, a.temperature, a.uniforms = P(256), 1, 100, 1.0, P(256)
        a.draft, a.draft_len, a.accept_len, a.next_token = P(256), P(256), P(256), P(256)
        a.workspace, a.workspace_bytes = P(256), pk.pldp_verify_sample_draft_workspace_size(2, 4, 100)
        return a

    def call(a):
        return lib.pldp_verify_sample_draft(ctypes.byref(a), None)

    assert lib.pldp_verify_sample_draft(None, None) == pk.PLDP_ERR_INVALID_ARG
    a = block(); a.next.index = None
    assert call(a) == pk.PLDP_ERR_INVALID_ARG and "index" in pk.pldp_last_error()
    for T in (0.0, -1.0, float("inf"), float("nan")):
        a = block(); a.temperature = T
        assert call(a) == pk.PLDP_ERR_INVALID_ARG and "temperature" in pk.pldp_last_error()
    a = block(); a.uniforms = None
    assert call(a) == pk.PLDP_ERR_INVALID_ARG and "null" in pk.pldp_last_error()
    a = block(); a.dtype = 7
    assert call(a) == pk.PLDP_ERR_UNSUPPORTED
    a = block(); a.next.ngram_max = 0
    assert call(a) == pk.PLDP_ERR_INVALID_ARG and "verify_sample_draft" in pk.pldp_last_error()
    a = block(); a.workspace_bytes = pk.pldp_verify_sample_draft_workspace_size(2, 4, 100) - 16
    assert call(a) == pk.PLDP_ERR_INVALID_ARG and "workspace" in pk.pldp_last_error()
    a = block(); a.next.B = 0
    assert call(a) == pk.PLDP_OK
    assert pk.pldp_verify_sample_draft_workspace_size(2, 4, 100) >= pk.pldp_verify_sample_workspace_size(2, 4, 100)


def test_binding_checks_element_counts_and_shapes():
    """The binding passes raw pointers, so it refuses, before any call, a buffer
    with fewer elements than the call touches, a status buffer that is not 4-byte
    words, an ids tensor with too few rows, and a T_cap beyond the ids rows."""
    import torch
    with pytest.raises(ValueError, match="needs 4 elements"):
        pk._dense(torch.zeros(3, dtype=torch.int32), "x", torch.int32, n=4)
    with pytest.raises(ValueError, match="int32 or uint32"):
        pk._dense(torch.zeros(4, dtype=torch.int64), "status", pk._WORD, n=4)
    with pytest.raises(ValueError, match="contiguous"):
        pk._dense(torch.zeros((4, 4), dtype=torch.int32)[:, :2], "x", torch.int32, n=4)
    with pytest.raises(ValueError, match="rows"):
        pk._rows(torch.zeros((2, 5), dtype=torch.int32), "ids", B=3)
    with pytest.raises(ValueError, match="T_cap"):
        pk._rows(torch.zeros((2, 5), dtype=torch.int32), "ids", T_cap=6)
    with pytest.raises(ValueError, match="unit inner stride"):
        pk._rows(torch.zeros((5, 2), dtype=torch.int32).t(), "ids")
    # a tensor of the right size still has to be on the device
    with pytest.raises(ValueError, match="CUDA"):
        pk._dense(torch.zeros(4, dtype=torch.int32), "x", torch.int32, n=4)


def _c_kind(decl):
    """('ptr',) for a pointer, (kind, bytes) for a scalar C parameter or return type."""
    decl = re.sub(r"/\*.*?\*/", "", decl).strip()
    if "*" in decl:
        return ("ptr",)
    words = [w for w in re.split(r"\s+", decl) if w not in ("const", "unsigned", "signed")]
    base = words[0]
    scalar = {"int": ("int", 4), "int32_t": ("int", 4), "uint32_t": ("int", 4), "int64_t": ("int", 8),
              "size_t": ("int", 8), "float": ("float", 4), "double": ("float", 8),
              "pldp_dtype": ("int", 4), "pldp_agg": ("int", 4), "pldp_status": ("int", 4)}
    return scalar[base]


def _ctypes_kind(t):
    if t is None:
        return None
    if t in (ctypes.c_void_p, ctypes.c_char_p) or issubclass(t, ctypes._Pointer):
        return ("ptr",)
    if t in (ctypes.c_float, ctypes.c_double):
        return ("float", ctypes.sizeof(t))
    return ("int", ctypes.sizeof(t))


def test_binding_signatures_match_the_header(so):
    """Every call's ctypes argtypes and restype in the binding agree with the
    prototype in include/pldp.h: the same number of parameters, a pointer where the
    header has one, and integer and floating scalars of the header's width."""
    src = re.sub(r"//[^\n]*", "", open(HEADER).read())
    protos = re.findall(r"PLDP_API\s+([\w\s\*]+?)\b(pldp_\w+)\s*\(([^;]*?)\)\s*;", src, flags=re.S)
    assert len(protos) == len(declared_symbols())
    lib = pk._load()
    for ret, name, params in protos:
        params = re.sub(r"/\*.*?\*/", "", params, flags=re.S).strip()
        want = [] if params in ("", "void") else [_c_kind(re.sub(r"\b\w+\s*$", "", p.strip()) or p)
                                                  for p in params.split(",")]
        fn = getattr(lib, name)
        got = [_ctypes_kind(t) for t in (fn.argtypes or [])]
        assert got == want, (name, got, want)
        want_ret = ("ptr",) if "*" in ret else _c_kind(ret)
        assert _ctypes_kind(fn.restype) == want_ret, (name, fn.restype, want_ret)


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    """Without libpldp.so every call raises: there is no CPU path to fall back to."""
    import torch
    monkeypatch.setattr(pk._build, "LIB", str(tmp_path / "libpldp.so"))
    monkeypatch.setattr(pk, "_lib", None)
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        pk.pldp_version()
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        pk.pldp_verify_workspace_size(2, 4, 100)
    x = torch.zeros((2, 8), dtype=torch.int32)
    with pytest.raises((RuntimeError, ValueError)):
        pk.pldp_find_candidates(x, torch.zeros(2, dtype=torch.int32), 1, 3, torch.zeros((2, 4), dtype=torch.int32),
                                torch.zeros(2, dtype=torch.int32), torch.zeros(2, dtype=torch.int32))
