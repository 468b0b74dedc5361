"""Seeded synthetic inputs for the DeLS-Spec per-block drafting path.

This module produces DATA only: random weights, logits and token counts with
the shapes and value distributions of the workloads the drafting path is run
on. It contains none of the method's arithmetic (no fusion, no softmax, no
argmax, no local-head forward, no prior estimation), so both the CPU oracle
and the CUDA path may consume what it returns without sharing any method code.

Everything is drawn from torch generators seeded per workload, on the device
the caller asks for (CPU for small cases, CUDA for the full-size ones, where
CPU generation of ~1e9 normals would dominate the test time). Tensors come
back as float32, bfloat16 or int64 torch tensors.

Workloads (shapes follow the paper's Qwen3 settings, Section 5.1, and the
local-head dimensions of Table 7):

* ``tiny``            B=1,  n=8,  V=1024,   1-layer MLP head over the last 2
                       drafted tokens (d=128, GELU), fp32 weights N(0, 0.02).
* ``qwen3_0p6b``      B=1,  n=16, V=151936, 2-layer MLP head over the last 4
                       drafted tokens (hidden 1024), bf16 weights N(0, 0.02),
                       fp32 logits.
* ``qwen3_4b``        B=8,  n=16, V=151936, 1-layer causal transformer head
                       (d=2560, 8 heads, FFN 10240), bf16 weights, fp32 logits.
* ``qwen3_8b_batched`` B=64, n=16, V=151936, GRU head of Appendix A
                       (embedding 4096, GRU 1024, rank 256), bf16 weights
                       N(0, 0.02), bf16 logits N(0, 3) plus a Zipf(1.1) bias.

The long-context logits stand in for the DFlash drafter's output and the
target logits for the target model's verification forward; neither model's
checkpoints are available, so both are synthetic (target = long + noise).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, Optional

import torch

__all__ = [
    "HeadSpec",
    "Workload",
    "WORKLOADS",
    "stress",
    "with_sizes",
    "make_inputs",
    "make_head_weights",
    "make_long_logits",
    "make_target_logits",
    "make_counts",
    "make_corpus",
    "CORPUS_TOKENS",
    "make_combine_inputs",
    "make_planted_verify",
    "sweep_points",
]

_DT = {"f32": torch.float32, "bf16": torch.bfloat16}


@dataclasses.dataclass(frozen=True)
class HeadSpec:
    """Shape of a local head (the short-context expert)."""

    kind: str                 # 'gru' | 'mlp' | 'xfmr' | 'markov'
    wdtype: str               # 'f32' | 'bf16'
    d_model: int              # embedding width
    d_hidden: int             # GRU state / MLP hidden / transformer FFN width
    d_rank: int               # width of the vector fed to the vocab projection
    window: int = 0           # MLP: number of previous drafted tokens
    n_layers: int = 1         # MLP: 1 or 2 hidden layers
    n_heads: int = 0          # transformer attention heads
    max_pos: int = 0          # transformer: rows of the position table


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int
    n: int
    V: int
    logit_dtype: str          # 'f32' | 'bf16'
    head: Optional[HeadSpec]
    weight: float             # combination weight w; alpha = beta = w
    long_std: float = 3.0     # std of the long-context logits
    target_noise: float = 1.0 # std of the target-minus-long noise
    zipf: float = 0.0         # Zipf exponent of the per-token logit bias (0: none)
    weight_std: Optional[float] = 0.02   # None: fan-in scaled (1/sqrt(fan_in))
    emb_std: float = 0.02
    seed: int = 0

    @property
    def alpha(self) -> float:
        return self.weight

    @property
    def beta(self) -> float:
        return self.weight


WORKLOADS: Dict[str, Workload] = {
    "tiny": Workload(
        "tiny", B=1, n=8, V=1024, logit_dtype="f32",
        head=HeadSpec("mlp", "f32", d_model=128, d_hidden=128, d_rank=128, window=2, n_layers=1),
        weight=0.5, long_std=2.0, target_noise=0.5, seed=0),
    "qwen3_0p6b": Workload(
        "qwen3_0p6b", B=1, n=16, V=151936, logit_dtype="f32",
        head=HeadSpec("mlp", "bf16", d_model=1024, d_hidden=1024, d_rank=1024, window=4, n_layers=2),
        weight=0.5, seed=1),
    "qwen3_4b": Workload(
        "qwen3_4b", B=8, n=16, V=151936, logit_dtype="f32",
        head=HeadSpec("xfmr", "bf16", d_model=2560, d_hidden=10240, d_rank=2560, n_heads=8, max_pos=16),
        weight=0.5, seed=2),
    "qwen3_8b_batched": Workload(
        "qwen3_8b_batched", B=64, n=16, V=151936, logit_dtype="bf16",
        head=HeadSpec("gru", "bf16", d_model=4096, d_hidden=1024, d_rank=256),
        weight=0.3, zipf=1.1, seed=3),
}


def stress(w: Workload) -> Workload:
    """Same shapes, fan-in-scaled weights and unit embeddings.

    With N(0, 0.02) weights the short logits are of order 1e-3 and never move
    a token; this variant makes them of order one so the local head matters.
    """
    return dataclasses.replace(w, name=w.name + "_stress", weight_std=None,
                               emb_std=1.0, seed=100 + w.seed)


def with_sizes(w: Workload, **kw) -> Workload:
    """Copy of a workload with some sizes replaced (e.g. V, B, n, head dims)."""
    head_kw = {k[5:]: kw.pop(k) for k in list(kw) if k.startswith("head_")}
    head = dataclasses.replace(w.head, **head_kw) if (w.head is not None and head_kw) else w.head
    return dataclasses.replace(w, head=head, **kw)


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _normal(shape, std, g, device, dtype) -> torch.Tensor:
    x = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        x.mul_(std)
    return x.to(_DT[dtype]) if dtype != "f32" else x


def _wstd(w: Workload, fan_in: int) -> float:
    return w.weight_std if w.weight_std is not None else 1.0 / math.sqrt(fan_in)


def make_head_weights(w: Workload, device="cpu") -> Dict[str, torch.Tensor]:
    """Weights of the local head, row-major [out, in] like a Linear layer."""
    h = w.head
    g = _gen(w.seed * 7919 + 11, device)
    dt = h.wdtype
    out: Dict[str, torch.Tensor] = {}
    if h.kind == "gru":
        out["emb"] = _normal((w.V, h.d_model), w.emb_std, g, device, dt)
        out["w_ih"] = _normal((3 * h.d_hidden, h.d_model), _wstd(w, h.d_model), g, device, dt)
        out["w_hh"] = _normal((3 * h.d_hidden, h.d_hidden), _wstd(w, h.d_hidden), g, device, dt)
        out["w_rank"] = _normal((h.d_rank, h.d_hidden), _wstd(w, h.d_hidden), g, device, dt)
        out["w_vocab"] = _normal((w.V, h.d_rank), _wstd(w, h.d_rank), g, device, dt)
    elif h.kind == "mlp":
        out["emb"] = _normal((w.V, h.d_model), w.emb_std, g, device, dt)
        fan = h.window * h.d_model
        out["w1"] = _normal((h.d_hidden, fan), _wstd(w, fan), g, device, dt)
        if h.n_layers == 2:
            out["w2"] = _normal((h.d_hidden, h.d_hidden), _wstd(w, h.d_hidden), g, device, dt)
        out["w_vocab"] = _normal((w.V, h.d_hidden), _wstd(w, h.d_hidden), g, device, dt)
    elif h.kind == "xfmr":
        d = h.d_model
        out["emb"] = _normal((w.V, d), w.emb_std, g, device, dt)
        out["pos"] = _normal((h.max_pos, d), w.emb_std, g, device, dt)
        for name in ("wq", "wk", "wv", "wo"):
            out[name] = _normal((d, d), _wstd(w, d), g, device, dt)
        out["w1"] = _normal((h.d_hidden, d), _wstd(w, d), g, device, dt)
        out["w2"] = _normal((d, h.d_hidden), _wstd(w, h.d_hidden), g, device, dt)
        out["w_vocab"] = _normal((w.V, d), _wstd(w, d), g, device, dt)
    elif h.kind == "markov":
        out["emb"] = _normal((w.V, h.d_rank), w.emb_std, g, device, dt)
        out["w_vocab"] = _normal((w.V, h.d_rank), _wstd(w, h.d_rank), g, device, dt)
    else:
        raise ValueError(f"unknown head kind {h.kind!r}")
    return out


def _zipf_rank(V: int, seed: int, device) -> torch.Tensor:
    """A seeded permutation pi: token v has frequency rank pi[v] (0 = most frequent)."""
    return torch.randperm(V, generator=_gen(seed * 31 + 5, "cpu")).to(device)


def make_long_logits(w: Workload, device="cpu") -> torch.Tensor:
    """Long-context (DFlash) logits [B, n, V]: N(0, long_std), plus a Zipf bias
    -zipf * ln(pi(v) + 1) when the workload asks for one."""
    g = _gen(w.seed * 7919 + 23, device)
    x = torch.randn(w.B, w.n, w.V, generator=g, device=device, dtype=torch.float32)
    x.mul_(w.long_std)
    if w.zipf:
        rank = _zipf_rank(w.V, w.seed, device).to(torch.float32)
        x.add_(torch.log1p(rank).mul_(-w.zipf))
    return x.to(_DT[w.logit_dtype]) if w.logit_dtype != "f32" else x


def make_target_logits(w: Workload, long: torch.Tensor, device="cpu") -> torch.Tensor:
    """Target logits [B, n+1, V]: rows 0..n-1 are the long logits plus
    N(0, target_noise); row n (the bonus row) is a fresh long-like row plus noise."""
    g = _gen(w.seed * 7919 + 37, device)
    B, n, V = long.shape
    t = torch.empty(B, n + 1, V, device=device, dtype=torch.float32)
    t[:, :n] = long.to(torch.float32)
    extra = torch.randn(B, V, generator=g, device=device, dtype=torch.float32).mul_(w.long_std)
    t[:, n] = extra
    t.add_(torch.randn(B, n + 1, V, generator=g, device=device, dtype=torch.float32).mul_(w.target_noise))
    return t.to(_DT[w.logit_dtype]) if w.logit_dtype != "f32" else t


def make_counts(w: Workload, total: float = 1e7) -> torch.Tensor:
    """Synthetic corpus token counts c[v] = floor(total * q(v)) with
    q(v) proportional to (pi(v) + 1)^(-1.1): a Zipf(1.1) unigram law over a
    seeded frequency ranking (the same ranking as the long-logit bias)."""
    rank = _zipf_rank(w.V, w.seed, "cpu").to(torch.float64)
    q = (rank + 1.0).pow(-1.1)
    q = q / q.sum()
    return torch.floor(q * total).to(torch.int64)


# Size of the synthetic training corpus the prior is estimated from: 2^28
# token positions (1.34 GB as int32 ids plus a byte mask), of the order of a
# ShareGPT-style chat corpus of ~100K conversations.
CORPUS_TOKENS = 1 << 28


def make_corpus(V: int, N: int, seed: int, device="cpu", chunk: int = 1 << 25):
    """A synthetic chat corpus of N token positions: (tokens int32 [N], loss_mask uint8 [N]).

    Ids follow the Zipf(1.1) law of ``make_counts`` over the same seeded
    frequency ranking, drawn by inverse-CDF lookup of uniform variates. The
    mask alternates user spans (mask 0, lengths uniform in [8, 256]) with
    assistant spans (mask 1, lengths uniform in [16, 768]), so about three
    quarters of the positions carry loss, as in supervised chat data.
    """
    if N < 0 or V <= 0:
        raise ValueError("need N >= 0 and V > 0")
    g = _gen(seed * 7919 + 71, device)
    by_rank = torch.argsort(_zipf_rank(V, seed, device))          # token id of each rank
    q = (torch.arange(V, device=device, dtype=torch.float64) + 1.0).pow(-1.1)
    cdf = torch.cumsum(q, 0)
    cdf = cdf / cdf[-1]
    tokens = torch.empty(N, dtype=torch.int32, device=device)
    for a in range(0, N, chunk):
        b = min(N, a + chunk)
        u = torch.rand(b - a, generator=g, device=device, dtype=torch.float64)
        r = torch.searchsorted(cdf, u).clamp_(max=V - 1)
        tokens[a:b] = by_rank[r].to(torch.int32)
    spans = 2 * (N // (2 * (8 + 16)) + 1)                         # enough spans to cover N
    lo = torch.tensor([8, 16], device=device).repeat(spans // 2)
    hi = torch.tensor([257, 769], device=device).repeat(spans // 2)
    lens = lo + (torch.rand(spans, generator=g, device=device) * (hi - lo).to(torch.float32)).long()
    lens = torch.minimum(lens, hi - 1)
    vals = torch.tensor([0, 1], dtype=torch.uint8, device=device).repeat(spans // 2)
    cum = torch.cumsum(lens, 0)
    k = int(torch.searchsorted(cum, torch.tensor([N], device=device)).item()) + 1
    mask = torch.repeat_interleave(vals[:k], lens[:k])[:N].contiguous()
    return tokens, mask


def make_inputs(w: Workload, device="cpu", target: bool = True) -> Dict[str, torch.Tensor]:
    """All inputs of one drafting + verification block for workload ``w``."""
    d: Dict[str, torch.Tensor] = {}
    d["long"] = make_long_logits(w, device)
    if target:
        d["target"] = make_target_logits(w, d["long"], device)
    d["counts"] = make_counts(w)
    if w.head is not None:
        d.update({"head." + k: v for k, v in make_head_weights(w, device).items()})
    return d


def make_combine_inputs(rows: int, V: int, dtype: str, seed: int, device="cpu",
                        std: float = 3.0) -> Dict[str, torch.Tensor]:
    """Independent long and short logit rows [rows, V] ~ N(0, std) for the
    combine-only path, plus Zipf counts for the prior."""
    g = _gen(seed * 7919 + 53, device)
    long = _normal((rows, V), std, g, device, dtype)
    short = _normal((rows, V), std, g, device, dtype)
    w = Workload("combine", B=rows, n=1, V=V, logit_dtype=dtype, head=None, weight=0.0, seed=seed)
    return {"long": long, "short": short, "counts": make_counts(w)}


def make_planted_verify(B: int, n: int, V: int, dtype: str, seed: int, device="cpu"):
    """Target logits with a planted, known argmax per row and draft tokens that
    match it for a chosen number of leading positions.

    Rows are N(0, 3) clamped to [-48, 48]; the planted token of each row gets
    the value 56, so it is that row's unique maximum by construction. Draft
    token j of row b equals the planted token for j < accept[b] and differs
    from it at j = accept[b] (when accept[b] < n). Returns (target [B, n+1, V],
    draft [B, n] int32, planted [B, n+1] int64, accept [B] int64).
    """
    g = _gen(seed * 7919 + 71, "cpu")
    t = torch.randn(B, n + 1, V, generator=g, dtype=torch.float32).mul_(3.0).clamp_(-48.0, 48.0)
    planted = torch.randint(0, V, (B, n + 1), generator=g)
    accept = torch.randint(0, n + 1, (B,), generator=g)
    if B >= 1:
        accept[0] = n                      # one row accepts the whole block
    if B >= 2:
        accept[1] = 0                      # one row rejects the first token
    t.scatter_(2, planted.unsqueeze(2), 56.0)
    draft = planted[:, :n].clone()
    shift = torch.randint(1, max(V, 2), (B, n), generator=g)
    for b in range(B):
        a = int(accept[b])
        if a < n:
            draft[b, a:] = (planted[b, a:n] + shift[b, a:]) % V
    t = t.to(_DT[dtype]) if dtype != "f32" else t
    return t.to(device), draft.to(torch.int32).to(device), planted, accept


def sweep_points():
    """The combine/verify sweep grid: B x n x V x dtype x w."""
    for V in (32000, 151936):
        for dtype in ("f32", "bf16"):
            for B in (1, 8, 32, 64, 128, 256):
                for n in (8, 16, 32):
                    for w in (0.0, 0.5, 1.0):
                        yield dict(B=B, n=n, V=V, dtype=dtype, weight=w)
