"""Seeded synthetic workloads for the PLD+ drafting + verification step.

This module only MAKES INPUTS.  It holds none of the method's arithmetic (no
candidate search, ranking, drafting or verification); both the CUDA path's
tests/benchmark and the CPU oracle consume what it produces.

The paper measures on public task datasets (summarization, code and text
editing; Sec. 5.1) that are not available here.  These generators stand in for
them with the structure that matters to PLD+: an output that copies spans of
its input.

Recipe (every config):
  * prompt tokens: uniform in [0, V).
  * output tokens: a sequence of segments; each segment is, with probability
    ``p_copy``, a span of length U[span_min, span_max] copied from the prompt
    at a uniform source offset s >= 1, else one uniform token.  ``p_copy`` is
    set so that the expected fraction of copied output tokens is the config's
    ``copy_frac``, unless ``p_copy_per_segment`` fixes it directly.
  * hidden rows: N(0, 1); for every copied output position p with source s,
    row p-1 is set to row s-1 plus N(0, 0.1^2) noise (the row that predicts a
    copied token resembles the row that predicted its source).  Source rows are
    prompt rows, which are never overwritten.
  * single-step configs end on a copied-span start, so that the planted source
    is the true continuation at the measured step.
  * attention rows of query t-1 (R = layers x heads): softmax over keys 0..t-1
    of N(0, 1) logits, +6 at the source of x_t in ``planted_heads`` heads of
    every layer; keys >= t are 0.  Held key-major by default (the R values of one
    key side by side, [B, T_cap, R] in memory, seen as [B, R, T_cap]).
  * target logits: N(0, 1); a planted row gets its chosen token set to
    (row max + 1), which makes that token the unique argmax.
  * bf16 tensors come from torch's bf16 generators (round-to-nearest-even casts
    where a value is computed in fp32).

Token structure uses numpy's PCG64 (identical on every machine); float tensors
use a torch.Generator on the requested device.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int
    prompt_len: int
    out_len: int
    V: int
    K: int
    copy_frac: float = 0.6
    span_min: int = 2
    span_max: int = 32
    p_copy_per_segment: Optional[float] = None
    ngram_min: int = 1
    ngram_max: int = 3
    d: Optional[int] = None          # hidden width (None: attention ranking only)
    h_dtype: str = "bf16"
    logits_dtype: str = "bf16"
    layers: int = 0                  # attention rows = layers * heads
    heads: int = 0
    planted_heads: int = 0
    planted_logit: float = 6.0
    attn_layout: str = "key"         # memory order of the attention rows: "key" (the R values of a key
                                     # side by side) or "head" (each row's keys side by side)
    accept: str = "uniform"          # "fixed:<n>", "uniform" (U{0..K}) or "ground_truth"
    steps: int = 1
    seed: int = 1000
    C_cap: int = 1024

    @property
    def T(self):
        return self.prompt_len + self.out_len

    @property
    def R(self):
        return self.layers * self.heads

    def t_cap(self, steps: Optional[int] = None) -> int:
        steps = self.steps if steps is None else steps
        return _round_up(self.T + steps * (self.K + 1), 8)

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


def _round_up(x, m):
    return (x + m - 1) // m * m


CONFIGS = {w.name: w for w in (
    # batch 1, one step: 384-token prompt + 128 output tokens (70% copied, spans 4-16),
    # V = 32000, max n-gram 3, K = 10, fp32 hidden [512, 4096], fp32 logits with the first
    # 6 draft tokens accepted.
    Workload("one_step_b1_ctx512", B=1, prompt_len=384, out_len=128, V=32000, K=10, copy_frac=0.7,
             span_min=4, span_max=16, d=4096, h_dtype="f32", logits_dtype="f32",
             accept="fixed:6", seed=1001),
    # batch 8, context 4096 (3072 + 1024, 60% copied, spans 2-32), V = 32000, bf16 hidden
    # [8, 4096, 4096], K = 10, bf16 logits with accept length U{0..10}.
    Workload("hidden_b8_ctx4k", B=8, prompt_len=3072, out_len=1024, V=32000, K=10, copy_frac=0.6,
             span_min=2, span_max=32, d=4096, seed=1002),
    # batch 64, context 16384 (12288 + 4096, 50% copied, spans 2-64), V = 32000, bf16 hidden
    # width 5120, K = 16, bf16 logits [64, 17, 32000].
    Workload("hidden_b64_ctx16k", B=64, prompt_len=12288, out_len=4096, V=32000, K=16, copy_frac=0.5,
             span_min=2, span_max=64, d=5120, seed=1003),
    # attention ranking: batch 32, context 8192 (6144 + 2048, 60% copied, spans 2-32),
    # bf16 attention rows [32, 4 layers, 32 heads, 8192] with mass planted on the copy
    # source in 8 heads per layer, K = 10, bf16 logits [32, 11, 128256].
    Workload("attention_b32_ctx8k", B=32, prompt_len=6144, out_len=2048, V=128256, K=10, copy_frac=0.6,
             span_min=2, span_max=32, layers=4, heads=32, planted_heads=8, seed=1004),
    # sustained decode loop: batch 128, context 32768 (24576 + 8192), 256 steps; the ground
    # truth copies prompt spans (2-32) with probability 0.6 per segment, else a uniform
    # token; bf16 hidden width 4096 and attention rows [4 layers x 32 heads] both ranked;
    # V = 128256, K = 12.
    Workload("decode_loop_b128_ctx32k", B=128, prompt_len=24576, out_len=8192, V=128256, K=12,
             p_copy_per_segment=0.6, span_min=2, span_max=32, d=4096, layers=4,
             heads=32, planted_heads=8, accept="ground_truth", steps=256, seed=1005),
)}


def torch_dtype(name):
    return {"f32": torch.float32, "bf16": torch.bfloat16}[name]


# ----------------------------------------------------------------------------
# token structure (numpy, machine independent)
# ----------------------------------------------------------------------------
def _p_copy(w: Workload) -> float:
    if w.p_copy_per_segment is not None:
        return w.p_copy_per_segment
    mean_span = 0.5 * (w.span_min + w.span_max)
    f = w.copy_frac
    return f / (mean_span * (1.0 - f) + f)


def token_streams(w: Workload, total_len: int, seed: Optional[int] = None,
                  end_on_span_start: bool = False):
    """Returns (tokens int32 [B, total_len], src int32 [B, total_len]) where
    src[b, p] is the prompt position copied to p (-1: not copied).  With
    ``end_on_span_start`` the position w.T-1 is forced to start a copied span whose
    source has at least K following prompt tokens."""
    rng = np.random.default_rng(w.seed if seed is None else seed)
    B, P = w.B, w.prompt_len
    tok = np.zeros((B, total_len), np.int32)
    src = np.full((B, total_len), -1, np.int32)
    p_copy = _p_copy(w)
    for b in range(B):
        tok[b, :P] = rng.integers(0, w.V, size=P)
        p = P
        while p < total_len:
            if rng.random() < p_copy:
                L = int(rng.integers(w.span_min, w.span_max + 1))
                s = int(rng.integers(1, P - L + 1))
                n = min(L, total_len - p)
                tok[b, p:p + n] = tok[b, s:s + n]
                src[b, p:p + n] = np.arange(s, s + n, dtype=np.int32)
                p += n
            else:
                tok[b, p] = rng.integers(0, w.V)
                p += 1
        if end_on_span_start:
            t = w.T - 1
            s = int(rng.integers(1, P - w.K - 1))
            tok[b, t] = tok[b, s]
            src[b, t] = s
    return tok, src


# ----------------------------------------------------------------------------
# float artifacts (torch, on any device)
# ----------------------------------------------------------------------------
def gen_hidden(w: Workload, src: np.ndarray, T_cap: int, device, gen: torch.Generator,
               out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Hidden rows [B, T_cap, d] of the workload's layer; planted as in the module doc."""
    dt = torch_dtype(w.h_dtype)
    B, d = w.B, w.d
    H = out if out is not None else torch.empty((B, T_cap, d), dtype=dt, device=device)
    for b in range(B):
        H[b].normal_(0.0, 1.0, generator=gen)
        pos = np.nonzero(src[b, :T_cap + 1] >= 0)[0]
        pos = pos[(pos >= 1) & (pos <= T_cap)]
        if pos.size == 0:
            continue
        rows = torch.from_numpy(pos - 1).to(device=device, dtype=torch.long)
        srows = torch.from_numpy(src[b, pos].astype(np.int64) - 1).to(device)
        for lo in range(0, rows.numel(), 65536):
            r, s = rows[lo:lo + 65536], srows[lo:lo + 65536]
            noise = torch.empty((r.numel(), d), dtype=torch.float32, device=device)
            noise.normal_(0.0, 0.1, generator=gen)
            H[b, r] = (H[b, s].float() + noise).to(dt)
    return H


def induction_rows(w: Workload) -> np.ndarray:
    """Indices (into the R = layers*heads rows) of the heads that carry the planted
    copy mass: a fixed seeded choice of ``planted_heads`` heads in every layer."""
    rng = np.random.default_rng(w.seed + 77)
    rows = []
    for l in range(w.layers):
        hs = np.sort(rng.choice(w.heads, w.planted_heads, replace=False))
        rows.extend(l * w.heads + hs)
    return np.asarray(rows, np.int32)


def empty_attention(w: Workload, T_cap: int, device) -> torch.Tensor:
    """An uninitialised [B, R, T_cap] bf16 attention tensor in the workload's memory
    order: key-major storage [B, T_cap, R] viewed as [B, R, T_cap], or head-major."""
    if w.attn_layout == "key":
        return torch.empty((w.B, T_cap, w.R), dtype=torch.bfloat16, device=device).transpose(1, 2)
    return torch.empty((w.B, w.R, T_cap), dtype=torch.bfloat16, device=device)


def gen_attention(w: Workload, seq_len: torch.Tensor, src_of_last: torch.Tensor, T_cap: int,
                  device, gen: torch.Generator, out: Optional[torch.Tensor] = None,
                  chunk: int = 8) -> torch.Tensor:
    """Attention rows of query t-1: [B, R, T_cap] bf16.  ``seq_len`` and
    ``src_of_last`` (the source of x_t, -1 if none) are device tensors [B]."""
    B, R = w.B, w.R
    A = out if out is not None else empty_attention(w, T_cap, device)
    planted = torch.zeros(R, dtype=torch.bool, device=device)
    planted[torch.from_numpy(induction_rows(w).astype(np.int64)).to(device)] = True
    keys = torch.arange(T_cap, device=device)
    for lo in range(0, B, chunk):
        hi = min(B, lo + chunk)
        lg = torch.empty((hi - lo, R, T_cap), dtype=torch.float32, device=device)
        lg.normal_(0.0, 1.0, generator=gen)
        t = (seq_len[lo:hi].long() - 1).clamp(min=0)
        s = src_of_last[lo:hi].long()
        hit = (keys[None, :] == s[:, None]) & (s[:, None] >= 0)           # [b, key]
        lg += w.planted_logit * (hit[:, None, :] & planted[None, :, None])
        lg.masked_fill_(keys[None, None, :] >= t[:, None, None], float("-inf"))
        lg = torch.softmax(lg, dim=-1)
        lg.nan_to_num_(0.0)                                                # t = 0: no keys
        A[lo:hi] = lg.to(torch.bfloat16)
        del lg
    return A


def gen_logits(w: Workload, targets: torch.Tensor, device, gen: torch.Generator,
               out: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Target logits [B, K+1, V]: N(0,1), and row (b, i) with targets[b, i] >= 0 gets
    that token planted as its unique argmax."""
    dt = torch_dtype(w.logits_dtype)
    B, K1, V = w.B, w.K + 1, w.V
    L = out if out is not None else torch.empty((B, K1, V), dtype=dt, device=device)
    L.normal_(0.0, 1.0, generator=gen)
    tg = targets.to(device=device, dtype=torch.long)
    sel = tg >= 0
    plant = (L.amax(dim=-1).float() + 1.0).to(dt)
    L.scatter_(2, tg.clamp(min=0)[..., None],
               torch.where(sel, plant, L.gather(2, tg.clamp(min=0)[..., None])[..., 0])[..., None])
    return L


# ----------------------------------------------------------------------------
# complete inputs
# ----------------------------------------------------------------------------
def single_step(w: Workload, device="cpu", seed: Optional[int] = None) -> dict:
    """All inputs of one decode step of a single-step config (a one-step workload or a variant).

    Returns a dict of tensors on ``device``: ids [B, T_cap] int32, seq_len [B] int32,
    H or None, A or None, logits; plus host numpy: src, expected_draft [B, K] (the
    prompt tokens after the planted source), planted_accept [B]."""
    seed = w.seed if seed is None else seed
    T_cap = w.t_cap(1)
    tok, src = token_streams(w, w.T, seed, end_on_span_start=True)
    ids = np.zeros((w.B, T_cap), np.int32)
    ids[:, :w.T] = tok
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    t = w.T - 1
    s_last = src[:, t]
    expected = np.stack([tok[b, s_last[b] + 1: s_last[b] + 1 + w.K] for b in range(w.B)])
    rng = np.random.default_rng(seed + 1)
    if w.accept.startswith("fixed:"):
        acc = np.full(w.B, int(w.accept.split(":")[1]), np.int64)
    else:
        acc = rng.integers(0, w.K + 1, size=w.B)
    targets = np.full((w.B, w.K + 1), -1, np.int64)
    for b in range(w.B):
        targets[b, :acc[b]] = expected[b, :acc[b]]
        if acc[b] < w.K:
            targets[b, acc[b]] = (expected[b, acc[b]] + 1 + rng.integers(0, w.V - 1)) % w.V
    out = dict(ids=torch.from_numpy(ids).to(device),
               seq_len=torch.full((w.B,), w.T, dtype=torch.int32, device=device),
               src=src, expected_draft=expected.astype(np.int32), planted_accept=acc.astype(np.int32),
               T_cap=T_cap, H=None, A=None)
    if w.d:
        out["H"] = gen_hidden(w, src, T_cap, device, gen)
    if w.R:
        out["A"] = gen_attention(w, out["seq_len"], torch.from_numpy(s_last).to(device), T_cap,
                                 device, gen)
        out["row_idx"] = induction_rows(w)
    out["logits"] = gen_logits(w, torch.from_numpy(targets), device, gen)
    return out


class DecodeLoop:
    """Sustained decode loop inputs (the decode loop or a variant).

    The ground-truth stream ``gt`` [B, T_cap] is fixed up front; the context starts as
    its first w.T tokens.  Before every step, ``step_inputs`` writes fresh attention
    rows for query t-1 and logits whose row i plants gt[b, seq_len + i] (the token
    greedy decoding emits there), reading the device-side seq_len.  Hidden rows for
    every position of the stream are generated once, since the rows a step appends are
    those of the ground-truth tokens."""

    def __init__(self, w: Workload, steps: int, device="cuda", seed: Optional[int] = None,
                 with_hidden: bool = True, with_attention: bool = True):
        self.w = w
        self.seed = w.seed if seed is None else seed
        self.steps = steps
        self.T_cap = w.t_cap(steps)
        self.device = device
        gt, src = token_streams(w, self.T_cap, self.seed)
        self.gt_host, self.src_host = gt, src
        self.gt = torch.from_numpy(gt).to(device)
        self.src = torch.from_numpy(src).to(device)
        ids = np.zeros_like(gt)
        ids[:, :w.T] = gt[:, :w.T]
        self.ids0 = torch.from_numpy(ids)
        self.ids = self.ids0.to(device)
        self.seq_len = torch.full((w.B,), w.T, dtype=torch.int32, device=device)
        self.gen = torch.Generator(device=device)
        self.gen.manual_seed(self.seed)
        self.H = gen_hidden(w, src, self.T_cap, device, self.gen) if (with_hidden and w.d) else None
        self.A = (empty_attention(w, self.T_cap, device)
                  if (with_attention and w.R) else None)
        self.logits = torch.empty((w.B, w.K + 1, w.V), dtype=torch_dtype(w.logits_dtype),
                                  device=device)
        self.row_idx = induction_rows(w) if w.R else None

    def reset(self):
        self.ids.copy_(self.ids0.to(self.device))
        self.seq_len.fill_(self.w.T)

    def step_inputs(self, step: int):
        """Regenerates A and logits for the current device-side state."""
        w = self.w
        self.gen.manual_seed(self.seed * 100003 + step)
        L = self.seq_len.long()
        idx = (L[:, None] + torch.arange(w.K + 1, device=self.device)[None]).clamp(max=self.T_cap - 1)
        targets = self.gt.gather(1, idx)
        if self.A is not None:
            s_last = self.src.gather(1, (L - 1).clamp(min=0)[:, None])[:, 0]
            gen_attention(w, self.seq_len, s_last, self.T_cap, self.device, self.gen, out=self.A)
        gen_logits(w, targets, self.device, self.gen, out=self.logits)

    def next_lengths(self, draft: torch.Tensor, draft_len: torch.Tensor) -> torch.Tensor:
        """The context lengths greedy verification of ``draft`` will leave: the
        logits plant gt[L + i] as row i's argmax, so n = the first i < draft_len with
        draft[i] != gt[L + i] (else draft_len), and L + n + 1 when that fits T_cap."""
        w = self.w
        L = self.seq_len.long()
        ar = torch.arange(w.K + 1, device=self.device)
        targets = self.gt.gather(1, (L[:, None] + ar[None]).clamp(max=self.T_cap - 1))
        d = draft_len.long().clamp(0, w.K)
        mism = (draft.long() != targets[:, :w.K]) | (ar[None, :w.K] >= d[:, None])
        n = torch.where(mism.any(dim=1), mism.int().argmax(dim=1), d)
        return torch.where(L + n + 1 <= self.T_cap, L + n + 1, L)

    def step_inputs_next(self, step: int, draft: torch.Tensor, draft_len: torch.Tensor):
        """Inputs of a step that verifies ``draft`` and drafts the next step in one
        call: logits for the current state, and attention rows for the query of the
        state verification will leave (the forward pass that produces this step's
        logits also produces those rows), from next_lengths."""
        w = self.w
        self.gen.manual_seed(self.seed * 100003 + step)
        L = self.seq_len.long()
        idx = (L[:, None] + torch.arange(w.K + 1, device=self.device)[None]).clamp(max=self.T_cap - 1)
        targets = self.gt.gather(1, idx)
        if self.A is not None:
            L_next = self.next_lengths(draft, draft_len)
            s_last = self.src.gather(1, (L_next - 1).clamp(min=0)[:, None])[:, 0]
            gen_attention(w, L_next.to(torch.int32), s_last, self.T_cap, self.device, self.gen, out=self.A)
        gen_logits(w, targets, self.device, self.gen, out=self.logits)
