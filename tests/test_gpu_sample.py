"""GPU parity of sampling verification (pldp_verify_sample) against the oracle.

The draws are decided in fp32 on the GPU and in fp64 in the oracle from the same
uniforms, so they may differ only where a uniform falls within rounding of a
boundary of the cumulative distribution; every other output (acceptance, bonus,
append, status) must then follow bit-exactly from the GPU's own draws."""
import numpy as np
import pytest
import torch
from scipy.special import softmax

import oracle
from tests._parity import host

pytestmark = pytest.mark.gpu
DEV = "cuda"
BOUNDARY_TOL = 2e-5


def i32(x):
    return torch.as_tensor(np.asarray(x, np.int32), device=DEV)


def _f64(logits):
    x = host(logits)
    return (oracle.bf16_to_f32(x) if x.dtype == np.uint16 else x).astype(np.float64)


def _valid_draw(row, T, u, y):
    """y is the inverse-CDF draw of some u' within BOUNDARY_TOL of u."""
    p = softmax(row / T)
    cdf = np.cumsum(p)
    lo = cdf[y - 1] if y > 0 else 0.0
    return p[y] > 0 and lo - BOUNDARY_TOL <= min(max(u, 0.0), 1.0 - 2 ** -24) < cdf[y] + BOUNDARY_TOL


def _run(logits, u, draft, dlen, T, ids=None, lens=None):
    B, K1, V = logits.shape
    K = K1 - 1
    ws = torch.empty(oracle_free_ws(B, K, V, logits.dtype), dtype=torch.uint8, device=DEV)
    out = {k: torch.full((B,), -7, dtype=torch.int32, device=DEV) for k in ("acc", "nxt", "kv")}
    sampled = torch.full((B, K1), -7, dtype=torch.int32, device=DEV)
    status = torch.zeros(B, dtype=torch.int32, device=DEV)
    import paper_2412_01447_gb300 as pk
    pk.pldp_verify_sample(logits, u, draft, dlen, out["acc"], out["nxt"], ws, temperature=T, sampled=sampled,
                          ids=ids, seq_len=lens, kv_keep_len=out["kv"] if lens is not None else None,
                          status=status)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}, sampled.cpu().numpy(), status.cpu().numpy().view(np.uint32)


def oracle_free_ws(B, K, V, dtype):
    import paper_2412_01447_gb300 as pk
    return pk.pldp_verify_sample_workspace_size(B, K, V, dtype)


@pytest.mark.parametrize("V,dtype", [(32000, torch.bfloat16), (128256, torch.bfloat16), (4096, torch.float32),
                                     (1001, torch.bfloat16), (999, torch.float32), (64, torch.bfloat16),
                                     (7, torch.bfloat16)])
@pytest.mark.parametrize("K,T", [(1, 1.0), (12, 0.7), (40, 1.3)])
def test_verify_sample_matches_oracle(lib, V, dtype, K, T):
    rng = np.random.default_rng(V + K)
    B, T_cap = 6, 96
    gen = torch.Generator(device=DEV).manual_seed(V * K)
    logits = (torch.randn((B, K + 1, V), generator=gen, device=DEV) * 2.5).to(dtype)
    u = rng.random((B, K + 1)).astype(np.float32)
    u[0, 0], u[1, 0], u[2, 0] = 0.0, 1.0, -0.5                  # clamped into [0, 1)
    l64 = _f64(logits)
    first = oracle.verify_sample(host(logits), u, np.zeros((B, K), np.int32), np.zeros(B, np.int32), T)["sampled"]
    draft = np.where(rng.random((B, K)) < 0.8, first[:, :K], rng.integers(0, V, size=(B, K))).astype(np.int32)
    dlen = rng.integers(0, K + 1, size=B).astype(np.int32)
    dlen[3] = K + 2                                              # clamped, flagged
    ids = rng.integers(0, V, size=(B, T_cap)).astype(np.int32)
    lens = rng.integers(1, T_cap - K - 1, size=B).astype(np.int32)
    lens[4] = T_cap - 1                                          # capacity
    ids_g, lens_g = i32(ids), i32(lens)
    g, ys, st = _run(logits, torch.from_numpy(u).to(DEV), i32(draft), i32(dlen), T, ids_g, lens_g)
    o = oracle.verify_sample(host(logits), u, draft, dlen, T)
    diff = np.argwhere(ys != o["sampled"])
    assert len(diff) <= max(2, ys.size // 500), diff
    for b, i in diff:
        assert _valid_draw(l64[b, i], T, float(u[b, i]), int(ys[b, i])), (b, i, ys[b, i], o["sampled"][b, i])
    # acceptance and bookkeeping follow from the GPU's draws exactly
    onehot = np.zeros((B, K + 1, V), np.float32)
    np.put_along_axis(onehot, ys[..., None].astype(np.int64), 1.0, axis=2)
    ids_o, lens_o = ids.copy(), lens.copy()
    e = oracle.verify_greedy(onehot, draft, dlen, ids=ids_o, seq_len=lens_o, kv_keep=True)
    assert np.array_equal(g["acc"], e["accept_len"]) and np.array_equal(g["nxt"], e["next_token"])
    assert np.array_equal(g["kv"], e["kv_keep_len"]) and np.array_equal(st, e["status"])
    assert np.array_equal(host(ids_g), ids_o) and np.array_equal(host(lens_g), lens_o)


def test_verify_sample_frequencies_are_softmax(lib):
    """Over a grid of uniforms the GPU's draws reproduce softmax(logits / T)."""
    V, N, T = 64, 8192, 0.8
    row = torch.linspace(-3, 2, V).to(torch.bfloat16)
    logits = row.expand(N, 2, V).contiguous().to(DEV)
    grid = (np.arange(N) + 0.5) / N
    u = torch.tensor(np.stack([grid, grid[::-1]], 1), dtype=torch.float32, device=DEV)
    _, ys, _ = _run(logits, u, torch.zeros((N, 1), dtype=torch.int32, device=DEV),
                    torch.zeros(N, dtype=torch.int32, device=DEV), T)
    p = softmax(oracle.bf16_to_f32(host(row)).astype(np.float64) / T)
    freq = np.bincount(ys[:, 0], minlength=V) / N
    assert np.abs(freq - p).max() <= 2.0 / N
    assert np.array_equal(np.bincount(ys[:, 1], minlength=V), np.bincount(ys[:, 0], minlength=V))


def test_verify_sample_low_temperature_is_greedy(lib):
    B, K, V = 16, 4, 32000
    gen = torch.Generator(device=DEV).manual_seed(3)
    logits = torch.randn((B, K + 1, V), generator=gen, device=DEV)
    logits[..., 123] += 8.0                                      # a clear maximum in every row
    u = torch.rand((B, K + 1), generator=gen, device=DEV) * 0.999
    _, ys, _ = _run(logits.to(torch.bfloat16), u, torch.zeros((B, K), dtype=torch.int32, device=DEV),
                    torch.zeros(B, dtype=torch.int32, device=DEV), 1e-3)
    assert (ys == 123).all()
