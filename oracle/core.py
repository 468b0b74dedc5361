"""Oracle core: prior, fusion, greedy decode, verification, statistics.

Test infrastructure only (see the package docstring). Plain fp64 numpy.
"""
from __future__ import annotations

import numpy as np


# ----------------------------------------------------------------------------
# data decoding (the oracle reads stored tensors itself; no shared helpers)
# ----------------------------------------------------------------------------

def to_f64(t) -> np.ndarray:
    """Exact float64 copy of a torch tensor or numpy array (f32, bf16, ints).

    bf16 is decoded from its bit pattern: the 16 stored bits are the upper
    half of an IEEE float32.
    """
    try:
        import torch
    except ImportError:  # pragma: no cover
        torch = None
    if torch is not None and isinstance(t, torch.Tensor):
        t = t.detach().cpu()
        if t.dtype == torch.bfloat16:
            bits = t.contiguous().view(torch.int16).numpy().view(np.uint16)
            return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        return t.numpy().astype(np.float64)
    return np.asarray(t, dtype=np.float64)


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round to bf16 (round-to-nearest-even) through float32; returns float64.

    This is the precision contract for activations that feed a bf16 product.
    """
    f = np.asarray(x, dtype=np.float32)
    if not np.all(np.isfinite(f)):
        raise ValueError("round_bf16: non-finite activation")
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    u = ((u + 0x7FFF + lsb) >> 16) << 16
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


# ----------------------------------------------------------------------------
# unigram prior (Appendix A, "Unigram Prior Estimation")
# ----------------------------------------------------------------------------

def count_masked_tokens(tokens, loss_mask, V: int):
    """c(v) = number of corpus positions t with loss_mask[t] == 1 and tokens[t] == v.

    Only loss-masked (assistant-response) tokens are counted. A masked
    position whose id lies outside [0, V) is not counted in c; it is reported
    separately. Returns (c as int64 [V], masked in-range total, masked
    out-of-range total).
    """
    t = np.asarray(tokens).reshape(-1).astype(np.int64)
    m = np.asarray(loss_mask).reshape(-1)
    if t.shape != m.shape:
        raise ValueError("tokens and loss_mask must have the same length")
    if V <= 0:
        raise ValueError("V must be positive")
    sel = t[m != 0]
    ok = (sel >= 0) & (sel < V)
    c = np.bincount(sel[ok], minlength=V).astype(np.int64)
    return c, int(ok.sum()), int((~ok).sum())


def log_prior(counts, lam: float = 1.0) -> np.ndarray:
    """l_P(v) = log( (c(v) + lambda) / sum_v' (c(v') + lambda) ), lambda = 1 by default."""
    c = to_f64(counts)
    if c.ndim != 1 or c.size == 0:
        raise ValueError("counts must be a non-empty vector")
    if np.any(c < 0) or lam <= 0:
        raise ValueError("counts must be >= 0 and lambda > 0")
    p = (c + lam) / np.sum(c + lam)
    return np.log(p)


# ----------------------------------------------------------------------------
# fusion and decode (Section 4.3 equation; Algorithm 1, Decode at T = 0)
# ----------------------------------------------------------------------------

def lse(x: np.ndarray) -> float:
    """log sum_v exp(x_v) for one row (textbook max-shifted form)."""
    x = np.asarray(x, dtype=np.float64)
    m = np.max(x)
    if m == -np.inf:
        raise ValueError("all entries are -inf")
    return float(m + np.log(np.sum(np.exp(x - m))))


def fuse(long, short, prior, alpha: float, beta: float) -> np.ndarray:
    """l = l_L + alpha * l_S - beta * l_P (Section 4.3). ``short``/``prior`` may be None
    (then that term is absent)."""
    out = np.array(long, dtype=np.float64, copy=True)
    if short is not None:
        out = out + alpha * np.asarray(short, dtype=np.float64)
    if prior is not None:
        out = out - beta * np.asarray(prior, dtype=np.float64)
    return out


def greedy_decode(l: np.ndarray):
    """Temperature-0 Decode(softmax(l)) of one row.

    Returns (x, logp, gap): x = argmax with the lowest index on exact ties,
    logp = log softmax(l)[x] = l[x] - LSE(l), gap = l[x] - max_{v != x} l[v]
    (+inf for a one-entry row).
    """
    l = np.asarray(l, dtype=np.float64)
    if np.any(np.isnan(l)) or np.any(l == np.inf):
        raise ValueError("non-finite logits")
    x = int(np.argmax(l))              # first occurrence of the maximum
    logp = float(l[x] - lse(l))
    if l.size == 1:
        gap = np.inf
    else:
        rest = np.concatenate([l[:x], l[x + 1:]])
        gap = float(l[x] - np.max(rest))
    return x, logp, gap


def combine_argmax(long, short, prior, alpha: float, beta: float):
    """Row-wise fuse + greedy decode of [rows, V] logits.

    Returns int64 tokens [rows], float64 logp [rows], float64 gap [rows].
    """
    L = to_f64(long)
    S = None if short is None else to_f64(short)
    P = None if prior is None else np.asarray(prior, dtype=np.float64)
    rows = L.shape[0]
    tok = np.zeros(rows, np.int64)
    lp = np.zeros(rows)
    gap = np.zeros(rows)
    for i in range(rows):
        f = fuse(L[i], None if S is None else S[i], P, alpha, beta)
        tok[i], lp[i], gap[i] = greedy_decode(f)
    return tok, lp, gap


# ----------------------------------------------------------------------------
# temperature-1 Decode (Algorithm 1, x_j ~ softmax(l^(j))) and its random numbers
# ----------------------------------------------------------------------------
# The random numbers come from Philox4x32-10, the counter-based generator of
# Salmon, Moraes, Dror and Shaw ("Parallel random numbers: as easy as 1, 2, 3",
# SC 2011): ten rounds on a counter of four 32-bit words under a key of two
# 32-bit words. A round multiplies words 0 and 2 by two fixed constants
# (32 x 32 -> 64-bit products), exchanges the words and folds the key into
# the high halves; the key is bumped by two Weyl constants between rounds.
# The drafting and verification kernels implement the same definition, so
# both sides draw identical uniforms from (seed, step, request, position,
# stream, vocabulary index).

PHILOX_M0, PHILOX_M1 = 0xD2511F53, 0xCD9E8D57
PHILOX_W0, PHILOX_W1 = 0x9E3779B9, 0xBB67AE85
STREAM_DRAFT, STREAM_ACCEPT, STREAM_RESIDUAL = 0, 1, 2
_M32 = np.uint64(0xFFFFFFFF)


def philox4x32_10(c0, c1, c2, c3, k0: int, k1: int):
    """Philox4x32-10 of the counter words (c0, c1, c2, c3) (integer arrays
    below 2^32, broadcast) under the key (k0, k1); returns the four output
    words as uint64 arrays holding 32-bit values."""
    x = [np.asarray(c, dtype=np.uint64) & _M32 for c in np.broadcast_arrays(c0, c1, c2, c3)]
    k0, k1 = np.uint64(k0 & 0xFFFFFFFF), np.uint64(k1 & 0xFFFFFFFF)
    s32 = np.uint64(32)
    for _ in range(10):
        p0 = x[0] * np.uint64(PHILOX_M0)          # < 2^64: exact in uint64
        p1 = x[2] * np.uint64(PHILOX_M1)
        x = [(p1 >> s32) ^ x[1] ^ k0, p1 & _M32, (p0 >> s32) ^ x[3] ^ k1, p0 & _M32]
        k0 = (k0 + np.uint64(PHILOX_W0)) & _M32
        k1 = (k1 + np.uint64(PHILOX_W1)) & _M32
    return x


def uniforms(seed: int, step: int, b: int, j: int, stream: int, v):
    """The uniform variates U(0, 1) of vocabulary indices v (array) for request
    b, position j and stream (0 drafting, 1 acceptance, 2 residual/bonus).

    Key (seed mod 2^32, seed div 2^32); counter (v div 4, step, b + 2^16 j +
    2^24 stream, 0); output word v mod 4 gives u = (floor(w / 2^9) + 1/2) /
    2^23, an exact float32 in [2^-24, 1 - 2^-24]. Needs 0 <= step < 2^32,
    0 <= b < 2^16 and 0 <= j < 2^8.
    """
    if not (0 <= step < 2 ** 32 and 0 <= b < 2 ** 16 and 0 <= j < 2 ** 8 and 0 <= stream < 4):
        raise ValueError("uniforms: step, request or position out of range")
    v = np.asarray(v, dtype=np.int64)
    seed &= 0xFFFFFFFFFFFFFFFF
    words = philox4x32_10((v >> 2).astype(np.uint64), np.uint64(step), np.uint64(b + (j << 16) + (stream << 24)),
                          np.uint64(0), seed & 0xFFFFFFFF, seed >> 32)
    w = np.select([(v & 3) == k for k in range(4)], words)
    return ((w >> np.uint64(9)).astype(np.float64) + 0.5) / float(1 << 23)


def gumbel(u):
    """Standard Gumbel variates g = -log(-log(u))."""
    return -np.log(-np.log(np.asarray(u, dtype=np.float64)))


def sample_decode(l, g):
    """Temperature-1 Decode of one row by the Gumbel-max rule: x = argmax(l + g)
    (lowest index on exact ties) is a draw from softmax(l) when g are i.i.d.
    standard Gumbel. Returns (x, logp = l[x] - LSE(l), key gap = k[x] - max_{v != x} k[v],
    LSE(l))."""
    l = np.asarray(l, dtype=np.float64)
    if np.any(np.isnan(l)) or np.any(l == np.inf):
        raise ValueError("non-finite logits")
    k = l + np.asarray(g, dtype=np.float64)
    x = int(np.argmax(k))
    z = lse(l)
    rest = np.concatenate([k[:x], k[x + 1:]])
    gap = float(k[x] - np.max(rest)) if rest.size else np.inf
    return x, float(l[x] - z), gap, z


def verify_sampled(draft, draft_logits, target, seed: int, step: int, request_ids=None):
    """Lossless speculative sampling (Leviathan et al. 2023; Chen et al. 2023)
    of a block drafted at temperature 1.

    draft [B, n] tokens; draft_logits [B, n, V] the logits each token was drawn
    from (row j: softmax gives q_j); target [B, n+1, V] (softmax gives p_j).
    For j = 0..n-1: accept x_j when u_j < p_j(x_j) / q_j(x_j), u_j the
    acceptance uniform of (b, j); at the first rejection the bonus token is
    drawn from the residual max(0, p_j - q_j) (normalised) by the Gumbel-max
    rule with the residual stream at position j; when all n are accepted it
    is drawn from p_n the same way at position n.

    ``request_ids``: the request index of each row for the random numbers
    (default 0..B-1).

    Returns (accept [B], bonus [B], info) with info["margin"][b] the distance
    |u - p/q| of the deciding test (the smallest over the accepted positions
    and the rejected one) and info["bonus_gap"][b] the key gap of the bonus draw.
    """
    D = np.asarray(draft, dtype=np.int64)
    Q = to_f64(draft_logits)
    T = to_f64(target)
    B, n = D.shape
    V = T.shape[2]
    if Q.shape != (B, n, V) or T.shape[:2] != (B, n + 1):
        raise ValueError("draft_logits must be [B, n, V] and target [B, n+1, V]")
    vidx = np.arange(V)
    accept = np.zeros(B, np.int64)
    bonus = np.zeros(B, np.int64)
    margin = np.full(B, np.inf)
    bonus_gap = np.zeros(B)
    for b in range(B):
        rid = b if request_ids is None else int(request_ids[b])
        a = n
        for j in range(n):
            p = np.exp(T[b, j] - lse(T[b, j]))
            q = np.exp(Q[b, j] - lse(Q[b, j]))
            x = D[b, j]
            u = float(uniforms(seed, step, rid, j, STREAM_ACCEPT, np.array([0]))[0])
            ratio = p[x] / q[x]
            margin[b] = min(margin[b], abs(u - ratio))
            if not u < ratio:
                a = j
                w = np.maximum(p - q, 0.0)
                with np.errstate(divide="ignore"):
                    key = np.log(w) + gumbel(uniforms(seed, step, rid, j, STREAM_RESIDUAL, vidx))
                break
        if a == n:
            key = T[b, n] + gumbel(uniforms(seed, step, rid, n, STREAM_RESIDUAL, vidx))
        accept[b] = a
        bonus[b] = int(np.argmax(key))
        rest = np.delete(key, bonus[b])
        bonus_gap[b] = float(key[bonus[b]] - np.max(rest)) if rest.size else np.inf
    return accept, bonus, {"margin": margin, "bonus_gap": bonus_gap}


# ----------------------------------------------------------------------------
# verification (Algorithm 1, greedy verification by one target forward)
# ----------------------------------------------------------------------------

def verify_greedy(draft, target):
    """Greedy verification of a drafted block against target logits.

    draft [B, n] tokens x_0..x_{n-1}; target [B, n+1, V] logits. Row j of the
    target gives its own choice t_j = argmax_v target[b, j, v] (lowest index on
    ties) for draft position j; row n is the bonus row. The accepted length a
    is the number of leading positions with x_j == t_j (0..n) and the bonus
    token is t_a. Returns (accept [B] int64, bonus [B] int64, t [B, n+1] int64).
    """
    D = np.asarray(draft, dtype=np.int64)
    T = to_f64(target)
    B, n = D.shape
    if T.shape[:2] != (B, n + 1):
        raise ValueError("target must be [B, n+1, V]")
    t = np.zeros((B, n + 1), np.int64)
    for b in range(B):
        for j in range(n + 1):
            row = T[b, j]
            if np.any(np.isnan(row)):
                raise ValueError("NaN target logits")
            t[b, j] = int(np.argmax(row))
    accept = np.zeros(B, np.int64)
    bonus = np.zeros(B, np.int64)
    for b in range(B):
        a = 0
        while a < n and D[b, a] == t[b, a]:
            a += 1
        accept[b] = a
        bonus[b] = t[b, a]
    return accept, bonus, t


# ----------------------------------------------------------------------------
# acceptance statistics (Appendix D)
# ----------------------------------------------------------------------------

def acceptance_rates(accept, n: int):
    """rate_i = P(acceptance length >= i), i = 1..n+1, and tau = E[length].

    The acceptance length counts the bonus token, L = a + 1, so rate_1 = 1
    (the first position is always produced). Returns (rates [n+1], tau).
    """
    a = np.asarray(accept, dtype=np.int64)
    if a.size == 0:
        raise ValueError("no blocks")
    L = a + 1
    rates = np.array([np.mean(L >= i) for i in range(1, n + 2)], dtype=np.float64)
    return rates, float(np.mean(L))


# ----------------------------------------------------------------------------
# exact factorisation (Section 4.1; proof in Appendix B)
# ----------------------------------------------------------------------------

def poe_factors(joint: np.ndarray):
    """Factors of p(x | y, z) for a joint table p[x, y, z] > 0.

    Returns (p_x_given_yz, poe, context, residual), each indexed [x, y, z]:
      poe      = p(x|y) p(x|z) / p(x)
      context  = p(y) p(z) / p(y, z)            (independent of x)
      residual = p(y, z | x) / (p(y|x) p(z|x))
    so that p(x|y,z) = poe * context * residual.
    """
    p = np.asarray(joint, dtype=np.float64)
    p = p / p.sum()
    px = p.sum(axis=(1, 2))
    py = p.sum(axis=(0, 2))
    pz = p.sum(axis=(0, 1))
    pxy = p.sum(axis=2)
    pxz = p.sum(axis=1)
    pyz = p.sum(axis=0)
    p_x_given_yz = p / pyz[None, :, :]
    p_x_given_y = pxy / py[None, :]
    p_x_given_z = pxz / pz[None, :]
    poe = p_x_given_y[:, :, None] * p_x_given_z[:, None, :] / px[:, None, None]
    context = (py[:, None] * pz[None, :] / pyz)[None, :, :] * np.ones_like(p)
    p_yz_given_x = p / px[:, None, None]
    p_y_given_x = pxy / px[:, None]
    p_z_given_x = pxz / px[:, None]
    residual = p_yz_given_x / (p_y_given_x[:, :, None] * p_z_given_x[:, None, :])
    return p_x_given_yz, poe, context, residual
