"""Oracle local heads and the per-block drafting loop (Algorithm 1).

Test infrastructure only (see the package docstring). Plain fp64 numpy; the
only library routines used are matrix products, exp/log/tanh and erf.

Every head maps a drafted prefix x_{0:j-1} (block tokens only, Section 3.2:
z_i = x_{k:i-1}) to a feature vector r, and l_S = W_vocab r (Appendix A). The
heads carry no state between blocks; within a block the GRU carries its
recurrent state along the prefix, the other heads recompute from the prefix.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, Optional

import numpy as np
from scipy.special import erf

from .core import (to_f64, round_bf16, fuse, greedy_decode, lse, sample_decode, gumbel, uniforms,
                   STREAM_DRAFT)


def _sigmoid(x):
    return 1.0 / (1.0 + np.exp(-x))


def _silu(x):
    return x * _sigmoid(x)


def _gelu(x):
    """GELU with the exact erf form: 0.5 x (1 + erf(x / sqrt 2))."""
    return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))


def _rmsnorm(x, eps=1e-6):
    """x / sqrt(mean(x^2) + eps) along the last axis (unit gain)."""
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)


class _Head:
    """Common part: weights as stored, the bf16 activation contract, W_vocab."""

    def __init__(self, weights: Dict[str, object], wdtype: str):
        self._raw = weights
        self.bf16 = (wdtype == "bf16")
        self._cache: Dict[str, np.ndarray] = {}

    def w(self, name) -> np.ndarray:
        if name not in self._cache:
            self._cache[name] = to_f64(self._raw[name])
        return self._cache[name]

    def emb_rows(self, name, tokens) -> np.ndarray:
        """Rows of an embedding table for the given token ids (decoded exactly)."""
        t = self._raw[name]
        try:
            import torch
            idx = torch.as_tensor(np.asarray(tokens, dtype=np.int64), device=t.device)
            return to_f64(t.index_select(0, idx))
        except (ImportError, AttributeError):  # numpy tables
            return to_f64(np.asarray(t)[np.asarray(tokens)])

    def act(self, x):
        """Activation fed to a matrix product: bf16-rounded for bf16 heads."""
        return round_bf16(x) if self.bf16 else x

    @property
    def V(self) -> int:
        return int(self._raw["w_vocab"].shape[0])

    def short_logits(self, feat: np.ndarray, chunk: int = 16384) -> np.ndarray:
        """l_S = W_vocab r for a batch of features r [B, d] -> [B, V].

        The product is taken over row blocks of W_vocab only to bound memory;
        every output entry is one complete dot product.
        """
        W = self._raw["w_vocab"]
        r = self.act(feat)
        B = r.shape[0]
        if "w_vocab" in self._cache:                       # already decoded whole (see w())
            return r @ self._cache["w_vocab"].T
        out = np.empty((B, self.V), dtype=np.float64)
        for v0 in range(0, self.V, chunk):
            Wc = to_f64(W[v0:v0 + chunk])
            out[:, v0:v0 + Wc.shape[0]] = r @ Wc.T
        return out


class GruHead(_Head):
    """RNN local head of Appendix A.

    e = E_tgt(x_{j-1}); one bias-free GRU layer in the PyTorch gate form with
    gate rows (r, z, n) in W_ih [3H, D] and W_hh [3H, H]:
        r_g = sigmoid(W_ir e + W_hr h)
        z   = sigmoid(W_iz e + W_hz h)
        c   = tanh(W_in e + r_g * (W_hn h))
        h'  = (1 - z) * c + z * h,          h_0 = 0
    then r = SiLU(W_rank h') and l_S = W_vocab r.
    """

    def __init__(self, weights, wdtype="bf16"):
        super().__init__(weights, wdtype)
        self.H = int(weights["w_hh"].shape[1])

    def init(self, B):
        return np.zeros((B, self.H), dtype=np.float64)

    def step(self, h, prev_tokens):
        H = self.H
        e = self.emb_rows("emb", prev_tokens)             # exact bf16 rows
        gi = self.act(e) @ self.w("w_ih").T                # [B, 3H]
        gh = self.act(h) @ self.w("w_hh").T                # [B, 3H]
        r_g = _sigmoid(gi[:, :H] + gh[:, :H])
        z = _sigmoid(gi[:, H:2 * H] + gh[:, H:2 * H])
        c = np.tanh(gi[:, 2 * H:] + r_g * gh[:, 2 * H:])
        h_new = (1.0 - z) * c + z * h
        feat = _silu(self.act(h_new) @ self.w("w_rank").T)
        return h_new, feat


class MlpHead(_Head):
    """Window MLP head (synthetic workloads): u = [E(x_{j-1}); ...; E(x_{j-W})],
    zero blocks for positions before the block start; h_1 = GELU(W_1 u);
    optionally h_2 = GELU(W_2 h_1); the last hidden vector is the feature."""

    def __init__(self, weights, wdtype, window, n_layers):
        super().__init__(weights, wdtype)
        self.window = int(window)
        self.n_layers = int(n_layers)
        self.D = int(weights["emb"].shape[1])

    def init(self, B):
        return [[] for _ in range(B)]          # per-row drafted prefix

    def step(self, hist, prev_tokens):
        B = len(hist)
        for b in range(B):
            hist[b].append(int(prev_tokens[b]))
        u = np.zeros((B, self.window * self.D))
        for b in range(B):
            for k in range(self.window):       # slot k holds x_{j-1-k}
                if len(hist[b]) - 1 - k >= 0:
                    tok = hist[b][len(hist[b]) - 1 - k]
                    u[b, k * self.D:(k + 1) * self.D] = self.emb_rows("emb", [tok])[0]
        h = _gelu(self.act(u) @ self.w("w1").T)
        if self.n_layers == 2:
            h = _gelu(self.act(h) @ self.w("w2").T)
        return hist, h


class XfmrHead(_Head):
    """One-layer causal pre-norm transformer over the block prefix (synthetic
    workload). Input t_p = E(x_p) + P[p] for p = 0..j-1; for the last position:
        a = RMSNorm(t),  q, k, v = W_q a, W_k a, W_v a  (per head, scale 1/sqrt(d_head))
        u = t_{j-1} + W_o attn(q_{j-1}, k_{0..j-1}, v_{0..j-1})
        y = u + W_2 GELU(W_1 RMSNorm(u));  feature = RMSNorm(y)
    RMSNorm has eps 1e-6 and unit gain; there are no biases.

    Precision: the head's own products take their activations unrounded
    (fp64 here); only the feature, which feeds the bf16 W_vocab product, is
    rounded to bf16 for bf16 heads (in short_logits)."""

    def __init__(self, weights, wdtype, n_heads):
        super().__init__(weights, wdtype)
        self.nh = int(n_heads)
        self.D = int(weights["emb"].shape[1])

    def init(self, B):
        return [[] for _ in range(B)]

    def step(self, hist, prev_tokens):
        B = len(hist)
        dh = self.D // self.nh
        feats = np.zeros((B, self.D))
        for b in range(B):
            hist[b].append(int(prev_tokens[b]))
            toks = hist[b]
            j = len(toks)
            t = self.emb_rows("emb", toks) + to_f64(self._raw["pos"][:j])
            a = _rmsnorm(t)
            q = a[-1] @ self.w("wq").T
            k = a @ self.w("wk").T
            v = a @ self.w("wv").T
            o = np.zeros(self.D)
            for hd in range(self.nh):
                sl = slice(hd * dh, (hd + 1) * dh)
                s = (k[:, sl] @ q[sl]) / math.sqrt(dh)
                p = np.exp(s - lse(s))
                o[sl] = p @ v[:, sl]
            u = t[-1] + o @ self.w("wo").T
            f = _gelu(_rmsnorm(u) @ self.w("w1").T)
            y = u + f @ self.w("w2").T
            feats[b] = _rmsnorm(y)
        return hist, feats


class MarkovHead(_Head):
    """Markov head of Appendix A: r = E_M(x_{i-1}), l_S = W_M r."""

    def init(self, B):
        return None

    def step(self, state, prev_tokens):
        return state, self.emb_rows("emb", prev_tokens)


def make_head(spec, weights):
    """Oracle head for a synth.HeadSpec and its weights (keys without 'head.')."""
    if spec.kind == "gru":
        return GruHead(weights, spec.wdtype)
    if spec.kind == "mlp":
        return MlpHead(weights, spec.wdtype, spec.window, spec.n_layers)
    if spec.kind == "xfmr":
        return XfmrHead(weights, spec.wdtype, spec.n_heads)
    if spec.kind == "markov":
        return MarkovHead(weights, spec.wdtype)
    raise ValueError(spec.kind)


@dataclasses.dataclass
class DraftResult:
    tokens: np.ndarray        # [B, n] the oracle's own greedy tokens (or the forced ones)
    logp: np.ndarray          # [B, n] log softmax(l^(j))[x_j] for the oracle's own argmax
    gap: np.ndarray           # [B, n] top-1 minus top-2 fused value
    argmax: np.ndarray        # [B, n] argmax of the fused logits at each position
    fused_at: Optional[np.ndarray] = None   # [B, n] fused value at the forced token
    fused_max: Optional[np.ndarray] = None  # [B, n] maximum fused value (forced mode)
    logp_at: Optional[np.ndarray] = None    # [B, n] log softmax at the forced token
    short_rows: Optional[Dict] = None       # {(b, j): l_S row} when requested
    lse: Optional[np.ndarray] = None        # [B, n] LSE of the fused row (temperature 1)
    fused: Optional[np.ndarray] = None      # [B, n, V] fused rows (temperature 1, keep_fused)


def draft_block(head, long, prior, alpha, beta, forced=None, keep_short=(), sample=None, keep_fused=False,
                request_ids=None):
    """Algorithm 1 for one block of B independent rows, at temperature 0
    (``sample=None``: Decode = argmax) or temperature 1 (``sample=(seed,
    step)``: Decode draws x_j from softmax(l^(j)) by the Gumbel-max rule,
    x_j = argmax(l^(j) + g), g the drafting-stream Gumbel variates of (b, j);
    ``gap`` and the forced-mode values then refer to the keys l + g).
    ``request_ids``: the request index of each row for the random numbers
    (default 0..B-1), so that a subset of a batch draws its own variates.

    long [B, n, V] long-context logits; prior [V] log unigram prior.
    Position 0: x_0 = argmax l_L^(0) (no local head, no prior term).
    Position j >= 1: l_S^(j) = head(x_{0:j-1}); l^(j) = l_L^(j) + alpha l_S^(j)
    - beta l_P; x_j = argmax l^(j).
    ``alpha`` / ``beta``: one weight for every position, or a sequence of n
    per-position weights (alpha_j, beta_j; entry 0 is unused) — the
    position-dependent weights whose learned values Appendix C reports.

    ``forced`` [B, n]: use these tokens as the drafted prefix instead of the
    oracle's own choices (to re-check a device run position by position after
    an argmax tie flipped a token). ``keep_short``: (b, j) pairs whose l_S row
    is returned for inspection.
    """
    L = long
    B, n, V = L.shape
    P = np.asarray(prior, dtype=np.float64)
    a_j = np.broadcast_to(np.asarray(alpha, dtype=np.float64), (n,)) if np.ndim(alpha) else np.full(n, float(alpha))
    b_j = np.broadcast_to(np.asarray(beta, dtype=np.float64), (n,)) if np.ndim(beta) else np.full(n, float(beta))
    tokens = np.zeros((B, n), np.int64)
    amax = np.zeros((B, n), np.int64)
    logp = np.zeros((B, n))
    gap = np.zeros((B, n))
    fused_at = np.zeros((B, n)) if forced is not None else None
    fused_max = np.zeros((B, n)) if forced is not None else None
    logp_at = np.zeros((B, n)) if forced is not None else None
    forced = None if forced is None else np.asarray(forced, dtype=np.int64)
    kept = {}
    lse_out = np.zeros((B, n)) if sample is not None else None
    fused_out = np.zeros((B, n, V)) if (sample is not None and keep_fused) else None
    vidx = np.arange(V)

    def row_long(b, j):
        return to_f64(L[b, j])

    def record(b, j, f):
        if sample is None:
            x, lp, g = greedy_decode(f)
            key = f
        else:
            rid = b if request_ids is None else int(request_ids[b])
            gv = gumbel(uniforms(sample[0], sample[1], rid, j, STREAM_DRAFT, vidx))
            x, lp, g, z = sample_decode(f, gv)
            key = f + gv
            lse_out[b, j] = z
            if fused_out is not None:
                fused_out[b, j] = f
        amax[b, j], logp[b, j], gap[b, j] = x, lp, g
        if forced is not None:
            xf = int(forced[b, j])
            tokens[b, j] = xf
            fused_at[b, j] = key[xf]
            fused_max[b, j] = key[x]
            logp_at[b, j] = f[xf] - lse(f)
        else:
            tokens[b, j] = x

    for b in range(B):
        record(b, 0, row_long(b, 0))
    state = head.init(B) if head is not None else None
    for j in range(1, n):
        prev = tokens[:, j - 1]
        state, feat = head.step(state, prev)
        S = head.short_logits(feat)
        for b in range(B):
            f = fuse(row_long(b, j), S[b], P, a_j[j], b_j[j])
            if (b, j) in keep_short:
                kept[(b, j)] = S[b].copy()
            record(b, j, f)
    return DraftResult(tokens, logp, gap, amax, fused_at, fused_max, logp_at, kept or None, lse_out, fused_out)
