"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test is chosen so that a plausible slip in the oracle (a dropped term, a
wrong sign or index, a transposed operand, an off-by-one in the verification
prefix) fails at least one of them. Library routines used as independent
references: scipy.special (logsumexp, log_softmax), torch CPU modules
(GRUCell, Linear, GELU, scaled_dot_product_attention, rms_norm).
"""
import itertools
import math
import os

import numpy as np
import pytest
import scipy.special as sps
import torch

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------- prior (App. A)

def test_prior_closed_forms():
    V = 7
    lp = oracle.log_prior(np.zeros(V, np.int64))
    np.testing.assert_allclose(lp, np.full(V, -math.log(V)), rtol=0, atol=1e-15)
    lp = oracle.log_prior(np.array([0, 1]))
    np.testing.assert_allclose(lp, [math.log(1 / 3), math.log(2 / 3)], atol=1e-15)
    lp = oracle.log_prior(np.array([4, 0, 10]), lam=2.0)
    np.testing.assert_allclose(lp, np.log(np.array([6, 2, 12]) / 20.0), atol=1e-15)


def test_masked_counts_brute_force():
    """c(v) counts only loss-masked positions; ids outside [0, V) are reported, not counted."""
    rng = np.random.default_rng(11)
    V, N = 37, 3001
    tok = rng.integers(-3, V + 4, size=N).astype(np.int32)
    mask = (rng.random(N) < 0.6).astype(np.uint8)
    mask[::7] = 2                                   # any nonzero byte carries loss
    c, n_in, n_out = oracle.count_masked_tokens(tok, mask, V)
    ref = [0] * V
    ref_in = ref_out = 0
    for t, m in zip(tok.tolist(), mask.tolist()):
        if m == 0:
            continue
        if 0 <= t < V:
            ref[t] += 1
            ref_in += 1
        else:
            ref_out += 1
    assert c.tolist() == ref and (n_in, n_out) == (ref_in, ref_out)
    assert c.dtype == np.int64 and c.shape == (V,)


def test_masked_counts_invariants():
    tok, mask = synth.make_corpus(1000, 20000, seed=3)
    tok, mask = tok.numpy(), mask.numpy()
    c, n_in, n_out = oracle.count_masked_tokens(tok, mask, 1000)
    assert n_out == 0 and n_in == int(mask.sum()) == int(c.sum())
    # the order of the corpus does not matter
    perm = np.random.default_rng(0).permutation(tok.size)
    c2, _, _ = oracle.count_masked_tokens(tok[perm], mask[perm], 1000)
    np.testing.assert_array_equal(c, c2)
    # counting a corpus in two pieces and adding gives the whole corpus's counts
    ca, _, _ = oracle.count_masked_tokens(tok[:7777], mask[:7777], 1000)
    cb, _, _ = oracle.count_masked_tokens(tok[7777:], mask[7777:], 1000)
    np.testing.assert_array_equal(ca + cb, c)
    # unmasked positions never count
    c0, z_in, z_out = oracle.count_masked_tokens(tok, np.zeros_like(mask), 1000)
    assert not c0.any() and z_in == z_out == 0
    # an empty corpus
    ce, e_in, e_out = oracle.count_masked_tokens(np.zeros(0, np.int32), np.zeros(0, np.uint8), 5)
    assert ce.tolist() == [0] * 5 and e_in == e_out == 0


def test_prior_from_a_balanced_corpus_is_uniform():
    """Every id loss-masked exactly k times: p0 is uniform whatever lambda is."""
    V, k = 50, 4
    tok = np.tile(np.arange(V, dtype=np.int32), k)
    tok = np.concatenate([tok, np.arange(V, dtype=np.int32)])     # unmasked tail
    mask = np.concatenate([np.ones(V * k, np.uint8), np.zeros(V, np.uint8)])
    c, _, _ = oracle.count_masked_tokens(tok, mask, V)
    assert c.tolist() == [k] * V
    for lam in (1.0, 0.25):
        np.testing.assert_allclose(oracle.log_prior(c, lam), np.full(V, -math.log(V)), atol=1e-15)


def test_synthetic_corpus_follows_its_zipf_law():
    """The corpus generator's masked frequencies follow q(v) ~ (pi(v) + 1)^-1.1 of make_counts."""
    w = synth.WORKLOADS["qwen3_8b_batched"]
    tok, mask = synth.make_corpus(w.V, 1 << 20, w.seed)
    c, n_in, _ = oracle.count_masked_tokens(tok.numpy(), mask.numpy(), w.V)
    assert 0.7 < n_in / tok.numel() < 0.8
    q = synth.make_counts(w, total=1.0 * n_in).numpy()        # floor(n_in * q(v))
    top = np.argsort(-q)[:20]
    np.testing.assert_allclose(c[top], q[top], rtol=0.05)


def test_prior_normalises_and_orders():
    c = synth.make_counts(synth.WORKLOADS["qwen3_8b_batched"])
    lp = oracle.log_prior(c)
    assert abs(np.exp(lp).sum() - 1.0) < 1e-12
    assert np.all(np.isfinite(lp))          # lambda = 1: no -inf entries
    cc = c.numpy()
    order = np.argsort(cc, kind="stable")
    assert np.all(np.diff(lp[order]) >= 0)  # monotone in the count


# ------------------------------------------------------- decode (Alg. 1, T = 0)

def test_lse_and_logsoftmax_against_scipy():
    rng = np.random.default_rng(0)
    x = rng.normal(0, 5, 1000)
    assert abs(oracle.lse(x) - sps.logsumexp(x)) < 1e-12
    tok, lp, gap = oracle.greedy_decode(x)
    ref = sps.log_softmax(x)
    assert tok == int(np.argmax(ref))
    assert abs(lp - ref[tok]) < 1e-12
    s = np.sort(x)
    assert abs(gap - (s[-1] - s[-2])) < 1e-15


def test_decode_ties_take_lowest_index_and_zero_gap():
    tok, lp, gap = oracle.greedy_decode(np.array([1.0, 3.0, 3.0, 2.0]))
    assert tok == 1 and gap == 0.0
    tok, lp, gap = oracle.greedy_decode(np.array([-np.inf, 0.5, -np.inf]))
    assert tok == 1 and abs(lp) < 1e-15 and gap == np.inf
    with pytest.raises(ValueError):
        oracle.greedy_decode(np.array([-np.inf, -np.inf]))
    with pytest.raises(ValueError):
        oracle.greedy_decode(np.array([0.0, np.nan]))


def test_fused_logprobs_normalise():
    rng = np.random.default_rng(1)
    L, S, P = rng.normal(0, 3, 500), rng.normal(0, 3, 500), np.log(rng.dirichlet(np.ones(500)))
    f = oracle.fuse(L, S, P, 0.3, 0.7)
    full = f - oracle.lse(f)
    assert abs(np.exp(full).sum() - 1.0) < 1e-12


def test_zero_weight_reproduces_dflash_argmax():
    d = synth.make_combine_inputs(rows=12, V=3000, dtype="bf16", seed=5)
    prior = oracle.log_prior(d["counts"])
    tok, lp, gap = oracle.combine_argmax(d["long"], d["short"], prior, 0.0, 0.0)
    L = oracle.to_f64(d["long"])
    np.testing.assert_array_equal(tok, np.argmax(L, axis=1))
    ref = sps.log_softmax(L, axis=1)
    np.testing.assert_allclose(lp, ref[np.arange(12), tok], atol=1e-12, rtol=0)


def test_row_and_prior_shifts_change_nothing():
    d = synth.make_combine_inputs(rows=6, V=2000, dtype="f32", seed=6)
    prior = oracle.log_prior(d["counts"])
    L = oracle.to_f64(d["long"])
    t0, lp0, g0 = oracle.combine_argmax(L, d["short"], prior, 0.5, 0.5)
    shift = np.arange(6)[:, None] * 17.25 - 40.0
    t1, lp1, g1 = oracle.combine_argmax(L + shift, d["short"], prior + 3.5, 0.5, 0.5)
    np.testing.assert_array_equal(t0, t1)
    np.testing.assert_allclose(lp0, lp1, atol=1e-9)
    np.testing.assert_allclose(g0, g1, atol=1e-9)


def test_alpha_beta_one_is_product_of_experts_in_probability_space():
    """At alpha = beta = 1 the fused softmax is p_L p_S / p_P renormalised (Eq. of Section 4.1)."""
    rng = np.random.default_rng(2)
    V = 64
    pL, pS, pP = (rng.dirichlet(np.ones(V) * 0.7) for _ in range(3))
    f = oracle.fuse(np.log(pL) + 2.0, np.log(pS) - 1.0, np.log(pP) + 0.25, 1.0, 1.0)
    q = np.exp(f - oracle.lse(f))
    ref = pL * pS / pP
    ref /= ref.sum()
    np.testing.assert_allclose(q, ref, rtol=1e-12, atol=1e-15)
    # a sign error on either weight would fail this
    g = oracle.fuse(np.log(pL), np.log(pS), np.log(pP), 1.0, -1.0)
    assert np.max(np.abs(np.exp(g - oracle.lse(g)) - ref)) > 1e-3


# --------------------------------------------------- factorisation (Sec. 4.1, App. B)

def test_three_factor_factorisation_is_exact():
    rng = np.random.default_rng(3)
    joint = rng.dirichlet(np.ones(4 * 3 * 4)).reshape(4, 3, 4)
    pxyz, poe, ctx, res = oracle.poe_factors(joint)
    np.testing.assert_allclose(poe * ctx * res, pxyz, rtol=1e-12)
    # the context factor does not depend on the candidate token
    assert np.max(np.abs(ctx - ctx[0:1])) < 1e-12
    np.testing.assert_allclose(pxyz.sum(axis=0), 1.0, rtol=1e-12)


def test_residual_is_one_under_conditional_independence_and_fusion_is_exact():
    rng = np.random.default_rng(4)
    X, Y, Z = 4, 3, 4
    px = rng.dirichlet(np.ones(X))
    py_x = rng.dirichlet(np.ones(Y), size=X)
    pz_x = rng.dirichlet(np.ones(Z), size=X)
    joint = px[:, None, None] * py_x[:, :, None] * pz_x[:, None, :]
    pxyz, poe, ctx, res = oracle.poe_factors(joint)
    np.testing.assert_allclose(res, 1.0, rtol=1e-12)
    pxy = joint.sum(axis=2)
    pxz = joint.sum(axis=1)
    for y in range(Y):
        for z in range(Z):
            lL = np.log(pxy[:, y] / pxy[:, y].sum())
            lS = np.log(pxz[:, z] / pxz[:, z].sum())
            lP = np.log(px)
            f = oracle.fuse(lL, lS, lP, 1.0, 1.0)
            np.testing.assert_allclose(np.exp(f - oracle.lse(f)), pxyz[:, y, z], rtol=1e-12)
            tok, _, _ = oracle.greedy_decode(f)
            assert tok == int(np.argmax(pxyz[:, y, z]))


# ------------------------------------------------------------ verification (Alg. 1)

def test_verify_planted_prefix():
    t, draft, planted, accept = synth.make_planted_verify(B=9, n=6, V=50, dtype="bf16", seed=7)
    a, bonus, tt = oracle.verify_greedy(draft, t)
    np.testing.assert_array_equal(tt, planted.numpy())
    np.testing.assert_array_equal(a, accept.numpy())
    np.testing.assert_array_equal(bonus, planted.numpy()[np.arange(9), accept.numpy()])
    assert a[0] == 6 and a[1] == 0


def test_verify_is_longest_matching_prefix_brute_force():
    rng = np.random.default_rng(8)
    B, n, V = 40, 5, 3
    T = rng.integers(-3, 3, size=(B, n + 1, V)).astype(np.float64)   # many exact ties
    draft = rng.integers(0, V, size=(B, n))
    a, bonus, t = oracle.verify_greedy(draft, T)
    for b in range(B):
        tb = [min(range(V), key=lambda v: (-T[b, j, v], v)) for j in range(n + 1)]
        best = max(k for k in range(n + 1) if all(draft[b, i] == tb[i] for i in range(k)))
        assert a[b] == best and bonus[b] == tb[best]


# ------------------------------------------------------- acceptance rates (App. D)

def _table6():
    rows = []
    with open(os.path.join(GOLDEN, "table6_acceptance_rates.txt")) as fh:
        for line in fh:
            if line.strip() and not line.startswith("#"):
                rows.append([float(x) for x in line.split()])
    return np.array(rows)


@pytest.mark.parametrize("col", [1, 2])
def test_acceptance_rates_reproduce_table6(col):
    tab = _table6()
    rates = tab[:, col] / 100.0                       # rate_1..rate_16
    N = 10000
    p_len = np.append(rates[:-1] - rates[1:], rates[-1])
    counts = np.rint(p_len * N).astype(int)
    assert counts.sum() == N
    lengths = np.repeat(np.arange(1, 17), counts)     # L = a + 1, L <= 16
    got, tau = oracle.acceptance_rates(lengths - 1, n=15)
    np.testing.assert_allclose(got, rates, atol=1e-12)
    assert abs(tau - rates.sum()) < 1e-12


# ------------------------------------------------------------ precision contract

def test_round_bf16_matches_torch_and_ties_to_even():
    rng = np.random.default_rng(9)
    x = rng.normal(0, 3, 10000).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(oracle.round_bf16(x), ref)
    # 1 + 2^-8 is halfway between 1 and 1 + 2^-7: ties go to the even mantissa (1.0)
    assert oracle.round_bf16(np.array([1.0 + 2 ** -8]))[0] == 1.0
    assert oracle.round_bf16(np.array([1.0 + 3 * 2 ** -8]))[0] == 1.0 + 2 ** -6


# ------------------------------------------------------------- local heads (App. A)

def _f32_weights(w):
    return {k[5:]: v for k, v in synth.make_inputs(w).items() if k.startswith("head.")}


def test_gru_head_matches_torch_grucell():
    w = synth.with_sizes(synth.stress(synth.WORKLOADS["qwen3_8b_batched"]), V=97, B=3, n=5,
                         head_wdtype="f32", head_d_model=24, head_d_hidden=16, head_d_rank=8)
    W = _f32_weights(w)
    head = oracle.GruHead(W, "f32")
    cell = torch.nn.GRUCell(24, 16, bias=False).double()
    with torch.no_grad():
        cell.weight_ih.copy_(W["w_ih"].double())
        cell.weight_hh.copy_(W["w_hh"].double())
    toks = [[5, 60, 7, 96], [0, 0, 1, 2], [33, 34, 35, 36]]
    h = head.init(3)
    ht = torch.zeros(3, 16, dtype=torch.float64)
    for j in range(4):
        prev = np.array([toks[b][j] for b in range(3)])
        h, feat = head.step(h, prev)
        e = W["emb"].double()[torch.as_tensor(prev)]
        ht = cell(e, ht)
        rt = torch.nn.functional.silu(ht @ W["w_rank"].double().T)
        np.testing.assert_allclose(h, ht.detach().numpy(), rtol=1e-12, atol=1e-14)
        np.testing.assert_allclose(feat, rt.detach().numpy(), rtol=1e-12, atol=1e-14)
    S = head.short_logits(feat)
    np.testing.assert_allclose(S, (rt @ W["w_vocab"].double().T).detach().numpy(), rtol=1e-12, atol=1e-13)


def test_gru_update_gate_saturated_keeps_state():
    """z -> 1 (huge positive z-gate weights): h' = h, so h stays at h_0 = 0."""
    w = synth.with_sizes(synth.stress(synth.WORKLOADS["qwen3_8b_batched"]), V=11, B=2, n=3,
                         head_wdtype="f32", head_d_model=8, head_d_hidden=4, head_d_rank=4)
    W = _f32_weights(w)
    W["w_ih"][4:8] = 0.0
    W["w_hh"][4:8] = 0.0
    W["emb"][:] = 1.0
    W["w_ih"][4:8] = 1e4             # z pre-activation = 8e4 > 0 for every input
    head = oracle.GruHead(W, "f32")
    h, _ = head.step(head.init(2), np.array([1, 2]))
    assert np.max(np.abs(h)) == 0.0


@pytest.mark.parametrize("layers", [1, 2])
def test_mlp_head_matches_torch(layers):
    w = synth.with_sizes(synth.stress(synth.WORKLOADS["qwen3_0p6b"]), V=50, B=2, n=6,
                         head_wdtype="f32", head_d_model=12, head_d_hidden=20, head_d_rank=20,
                         head_window=3, head_n_layers=layers)
    W = _f32_weights(w)
    head = oracle.MlpHead(W, "f32", 3, layers)
    seq = [[4, 9, 4, 0, 49], [1, 2, 3, 4, 5]]
    st = head.init(2)
    E = W["emb"].double()
    gelu = torch.nn.GELU(approximate="none")
    for j in range(5):
        st, feat = head.step(st, np.array([seq[0][j], seq[1][j]]))
        for b in range(2):
            parts = []
            for k in range(3):
                i = j - k
                parts.append(E[seq[b][i]] if i >= 0 else torch.zeros(12, dtype=torch.float64))
            u = torch.cat(parts)
            hh = gelu(u @ W["w1"].double().T)
            if layers == 2:
                hh = gelu(hh @ W["w2"].double().T)
            np.testing.assert_allclose(feat[b], hh.numpy(), rtol=1e-12, atol=1e-14)


def test_xfmr_head_matches_torch_causal_block():
    w = synth.with_sizes(synth.stress(synth.WORKLOADS["qwen3_4b"]), V=40, B=2, n=6,
                         head_wdtype="f32", head_d_model=16, head_d_hidden=32, head_d_rank=16,
                         head_n_heads=4, head_max_pos=6)
    W = _f32_weights(w)
    Wd = {k: v.double() for k, v in W.items()}
    head = oracle.XfmrHead(W, "f32", 4)
    seq = [[3, 39, 3, 0, 17], [8, 8, 8, 8, 8]]
    st = head.init(2)
    F = torch.nn.functional
    for j in range(5):
        st, feat = head.step(st, np.array([seq[0][j], seq[1][j]]))
        for b in range(2):
            toks = torch.as_tensor(seq[b][: j + 1])
            t = Wd["emb"][toks] + Wd["pos"][: j + 1]                     # [T, D]
            a = F.rms_norm(t, (16,), eps=1e-6)
            q, k, v = (a @ Wd[n].T for n in ("wq", "wk", "wv"))
            sh = lambda x: x.view(-1, 4, 4).transpose(0, 1)              # [heads, T, dh]
            o = F.scaled_dot_product_attention(sh(q), sh(k), sh(v), is_causal=True)
            o = o.transpose(0, 1).reshape(-1, 16)
            u = t + o @ Wd["wo"].T
            y = u + F.gelu(F.rms_norm(u, (16,), eps=1e-6) @ Wd["w1"].T) @ Wd["w2"].T
            ref = F.rms_norm(y, (16,), eps=1e-6)[-1]
            np.testing.assert_allclose(feat[b], ref.numpy(), rtol=1e-11, atol=1e-13)


def test_xfmr_head_bf16_contract_rounds_only_the_feature():
    """bf16 transformer head: the head's own products take unrounded
    activations (the same features as the torch float64 block above), and only
    the feature fed to W_vocab is rounded to bf16 (RNE)."""
    w = synth.with_sizes(synth.stress(synth.WORKLOADS["qwen3_4b"]), V=40, B=2, n=6,
                         head_d_model=16, head_d_hidden=32, head_d_rank=16, head_n_heads=4, head_max_pos=6)
    d = synth.make_inputs(w, target=False)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    assert W["wq"].dtype == torch.bfloat16
    Wd = {k: v.double() for k, v in W.items()}
    head = oracle.XfmrHead(W, "bf16", 4)
    st = head.init(2)
    F = torch.nn.functional
    seq = [[3, 39, 3, 0, 17], [8, 8, 8, 8, 8]]
    for j in range(5):
        st, feat = head.step(st, np.array([seq[0][j], seq[1][j]]))
        for b in range(2):
            toks = torch.as_tensor(seq[b][: j + 1])
            t = Wd["emb"][toks] + Wd["pos"][: j + 1]
            a = F.rms_norm(t, (16,), eps=1e-6)
            q, k, v = (a @ Wd[n].T for n in ("wq", "wk", "wv"))
            sh = lambda x: x.view(-1, 4, 4).transpose(0, 1)
            o = F.scaled_dot_product_attention(sh(q), sh(k), sh(v), is_causal=True).transpose(0, 1).reshape(-1, 16)
            u = t + o @ Wd["wo"].T
            y = u + F.gelu(F.rms_norm(u, (16,), eps=1e-6) @ Wd["w1"].T) @ Wd["w2"].T
            np.testing.assert_allclose(feat[b], F.rms_norm(y, (16,), eps=1e-6)[-1].numpy(), rtol=1e-11, atol=1e-13)
        S = head.short_logits(feat)
        r = torch.from_numpy(feat).float().bfloat16().double()
        np.testing.assert_allclose(S, (r @ Wd["w_vocab"].T).numpy(), rtol=1e-12, atol=1e-13)


def test_markov_head_is_embedding_times_vocab_matrix():
    w = synth.Workload("m", B=3, n=4, V=30, logit_dtype="f32",
                       head=synth.HeadSpec("markov", "f32", 0, 0, 6), weight=0.5, weight_std=None,
                       emb_std=1.0, seed=9)
    W = _f32_weights(w)
    head = oracle.MarkovHead(W, "f32")
    prev = np.array([0, 29, 7])
    _, feat = head.step(None, prev)
    S = head.short_logits(feat)
    ref = torch.nn.functional.embedding(torch.as_tensor(prev), W["emb"].double()) @ W["w_vocab"].double().T
    np.testing.assert_allclose(S, ref.numpy(), rtol=1e-12, atol=1e-14)


# ------------------------------------------------------- Algorithm 1 loop, brute force

@pytest.mark.parametrize("kind", ["mlp", "gru"])
def test_draft_block_brute_force_enumeration(kind):
    """V <= 8, n <= 4: among all V^n blocks exactly one has every x_j equal to the
    argmax of its own fused score given its own prefix, and the oracle returns it.
    The score is restated here from Algorithm 1: position 0 uses the long logits
    alone; positions j >= 1 add alpha * l_S(prefix) and subtract beta * l_P."""
    V, n, B = 6, 4, 2
    if kind == "mlp":
        base = synth.with_sizes(synth.stress(synth.WORKLOADS["tiny"]), V=V, B=B, n=n,
                                head_d_model=5, head_d_hidden=7, head_d_rank=7)
    else:
        base = synth.with_sizes(synth.stress(synth.WORKLOADS["qwen3_8b_batched"]), V=V, B=B, n=n,
                                head_wdtype="f32", head_d_model=5, head_d_hidden=4, head_d_rank=3,
                                logit_dtype="f32", zipf=0.0)
    d = synth.make_inputs(base, target=False)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = oracle.log_prior(d["counts"])
    alpha, beta = 1.3, 2.0          # large weights so that both terms move tokens
    L = oracle.to_f64(d["long"])
    res = oracle.draft_block(oracle.make_head(base.head, W), d["long"], prior, alpha, beta)
    for b in range(B):
        consistent = []
        for blk in itertools.product(range(V), repeat=n):
            ok = int(np.argmax(L[b, 0])) == blk[0]
            if ok:
                head = oracle.make_head(base.head, W)
                st = head.init(1)
                for j in range(1, n):
                    st, feat = head.step(st, np.array([blk[j - 1]]))
                    score = L[b, j] + alpha * head.short_logits(feat)[0] - beta * prior
                    if int(np.argmax(score)) != blk[j]:
                        ok = False
                        break
            if ok:
                consistent.append(blk)
        assert consistent == [tuple(res.tokens[b])]


def test_draft_block_position_zero_ignores_prior_and_head():
    base = synth.with_sizes(synth.stress(synth.WORKLOADS["tiny"]), V=40, B=3, n=3)
    d = synth.make_inputs(base, target=False)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = oracle.log_prior(d["counts"])
    r = oracle.draft_block(oracle.make_head(base.head, W), d["long"], prior, 5.0, 50.0)
    L = oracle.to_f64(d["long"])
    np.testing.assert_array_equal(r.tokens[:, 0], np.argmax(L[:, 0], axis=1))
    np.testing.assert_allclose(r.logp[:, 0], sps.log_softmax(L[:, 0], axis=1)[np.arange(3), r.tokens[:, 0]],
                               atol=1e-12)


def test_forced_prefix_mode_agrees_with_free_run():
    base = synth.with_sizes(synth.stress(synth.WORKLOADS["tiny"]), V=64, B=2, n=5)
    d = synth.make_inputs(base, target=False)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = oracle.log_prior(d["counts"])
    free = oracle.draft_block(oracle.make_head(base.head, W), d["long"], prior, 0.5, 0.5)
    forced = oracle.draft_block(oracle.make_head(base.head, W), d["long"], prior, 0.5, 0.5,
                                forced=free.tokens)
    np.testing.assert_array_equal(forced.argmax, free.tokens)
    np.testing.assert_allclose(forced.logp_at, free.logp, atol=1e-12)


# ------------------------------------------------- per-position weights (Appendix C)

def _learned_weights(n):
    """alpha_j, beta_j for j = 0..n-1 from the Appendix C table (positions 2..15
    are j = 1..14; later positions keep the last printed value; j = 0 unused)."""
    path = os.path.join(os.path.dirname(__file__), "golden", "appendix_c_learned_weights.txt")
    rows = [l.split() for l in open(path) if l.strip() and not l.startswith("#")]
    tab = {int(p): (float(a), float(b)) for p, a, b in rows}
    a = np.zeros(n)
    b = np.zeros(n)
    for j in range(1, n):
        a[j], b[j] = tab[min(j + 1, max(tab))]
    return a, b


def test_appendix_c_table_is_read_as_printed():
    a, b = _learned_weights(16)
    assert a[1] == 0.547 and b[1] == 0.512 and a[14] == 0.762 and b[12] == 0.617
    assert np.all(np.diff(a[1:]) >= 0)          # alpha grows with the position (Appendix C)


def test_constant_per_position_weights_equal_the_scalar_weight():
    base = synth.with_sizes(synth.stress(synth.WORKLOADS["tiny"]), V=64, B=3, n=6)
    d = synth.make_inputs(base, target=False)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = oracle.log_prior(d["counts"])
    r0 = oracle.draft_block(oracle.make_head(base.head, W), d["long"], prior, 0.7, 0.4)
    r1 = oracle.draft_block(oracle.make_head(base.head, W), d["long"], prior, np.full(6, 0.7), np.full(6, 0.4))
    np.testing.assert_array_equal(r0.tokens, r1.tokens)
    np.testing.assert_array_equal(r0.logp, r1.logp)


def test_zero_weight_at_one_position_reproduces_dflash_there():
    base = synth.with_sizes(synth.stress(synth.WORKLOADS["tiny"]), V=64, B=3, n=6)
    d = synth.make_inputs(base, target=False)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = oracle.log_prior(d["counts"])
    a, b = _learned_weights(6)
    a[3] = b[3] = 0.0
    r = oracle.draft_block(oracle.make_head(base.head, W), d["long"], prior, a, b)
    L = oracle.to_f64(d["long"])
    np.testing.assert_array_equal(r.tokens[:, 3], np.argmax(L[:, 3], axis=1))
    np.testing.assert_allclose(r.logp[:, 3], sps.log_softmax(L[:, 3], axis=1)[np.arange(3), r.tokens[:, 3]],
                               atol=1e-12)


def test_per_position_weights_brute_force_enumeration():
    """As the brute-force pin above, with a different (alpha_j, beta_j) at every
    position: exactly one block is greedy-consistent and the oracle returns it."""
    V, n, B = 6, 4, 2
    base = synth.with_sizes(synth.stress(synth.WORKLOADS["tiny"]), V=V, B=B, n=n,
                            head_d_model=5, head_d_hidden=7, head_d_rank=7)
    d = synth.make_inputs(base, target=False)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = oracle.log_prior(d["counts"])
    a = np.array([0.0, 2.1, 0.4, 1.6])
    b = np.array([0.0, 0.3, 2.5, 1.1])
    L = oracle.to_f64(d["long"])
    res = oracle.draft_block(oracle.make_head(base.head, W), d["long"], prior, a, b)
    for bb in range(B):
        consistent = []
        for blk in itertools.product(range(V), repeat=n):
            ok = int(np.argmax(L[bb, 0])) == blk[0]
            if ok:
                head = oracle.make_head(base.head, W)
                st = head.init(1)
                for j in range(1, n):
                    st, feat = head.step(st, np.array([blk[j - 1]]))
                    score = L[bb, j] + a[j] * head.short_logits(feat)[0] - b[j] * prior
                    if int(np.argmax(score)) != blk[j]:
                        ok = False
                        break
            if ok:
                consistent.append(blk)
        assert consistent == [tuple(res.tokens[bb])]


# ------------------------------------------- temperature 1 (Algorithm 1 Decode ~ softmax)

def _curand_host_philox(seed, offset, count):
    """`count` 32-bit outputs of cuRAND's host-side Philox4x32-10 generator
    (CURAND_RNG_PSEUDO_PHILOX4_32_10 = 161, default ordering) from `offset`."""
    import ctypes
    import os
    lib = None
    for name in (os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "lib64", "libcurand.so"),
                 "libcurand.so", "libcurand.so.10"):
        try:
            lib = ctypes.CDLL(name)
            break
        except OSError:
            continue
    if lib is None:
        pytest.skip("libcurand is not installed")
    gen = ctypes.c_void_p()
    assert lib.curandCreateGeneratorHost(ctypes.byref(gen), 161) == 0
    try:
        assert lib.curandSetPseudoRandomGeneratorSeed(gen, ctypes.c_ulonglong(seed)) == 0
        assert lib.curandSetGeneratorOffset(gen, ctypes.c_ulonglong(offset)) == 0
        out = np.zeros(count, dtype=np.uint32)
        assert lib.curandGenerate(gen, out.ctypes.data_as(ctypes.c_void_p), ctypes.c_size_t(count)) == 0
    finally:
        lib.curandDestroyGenerator(gen)
    return [int(x) for x in out]


@pytest.mark.parametrize("seed", [0, 1234, 0xFEDCBA9876543210, 2 ** 64 - 1])
def test_philox_matches_curands_host_philox4x32(seed):
    """Philox4x32-10 against the host generator of a library that implements
    the same published definition. That generator uses the key (seed mod
    2^32, seed div 2^32) and emits block k of four outputs from the counter
    (x0, x1, x2, 0) with x2 = k mod 2^16 and x0 + 2^32 x1 = k div 2^16; the
    cases reach every counter word the drafting path sets (word 3 is always
    0 there) with large and small values."""
    for x0, x1, x2 in [(0, 0, 0), (1, 0, 0), (0, 0, 1), (123456, 0, 17), (2 ** 32 - 1, 0, 65534),
                       (5, 3, 100), (77, 1, 65534), (2 ** 31 + 9, 11, 40000)]:
        k = x2 + (1 << 16) * (x0 + (x1 << 32))
        want = _curand_host_philox(seed, 4 * k, 8)
        got = oracle.philox4x32_10(np.array([x0, x0], dtype=np.uint64), x1, np.array([x2, x2 + 1], dtype=np.uint64),
                                   0, seed & 0xFFFFFFFF, seed >> 32)
        got = [int(got[w][i]) for i in range(2) for w in range(4)]
        assert got == want, (seed, x0, x1, x2)


def test_uniforms_reject_counter_fields_out_of_range():
    for args in ((1, 2 ** 32, 0, 0, 0), (1, 0, 2 ** 16, 0, 0), (1, 0, 0, 2 ** 8, 0), (1, -1, 0, 0, 0)):
        with pytest.raises(ValueError):
            oracle.uniforms(*args, np.arange(4))


def test_uniforms_lie_on_the_float32_grid_inside_the_unit_interval():
    u = oracle.uniforms(11, 2, 3, 4, oracle.STREAM_DRAFT, np.arange(4096))
    scaled = u * 2.0 ** 23 - 0.5
    assert np.all(scaled == np.round(scaled)) and np.all((u > 0) & (u < 1))
    assert np.all(u.astype(np.float32).astype(np.float64) == u)
    assert abs(u.mean() - 0.5) < 0.02
    # different streams, positions, requests and steps give different variates
    base = oracle.uniforms(11, 2, 3, 4, 0, np.arange(64))
    for args in ((11, 2, 3, 4, 1), (11, 2, 3, 5, 0), (11, 2, 4, 4, 0), (11, 3, 3, 4, 0), (12, 2, 3, 4, 0)):
        assert not np.array_equal(base, oracle.uniforms(*args, np.arange(64)))


def _chi2_p(counts, probs):
    from scipy.stats import chisquare
    counts = np.asarray(counts, dtype=np.float64)
    return chisquare(counts, counts.sum() * np.asarray(probs)).pvalue


def test_gumbel_max_draws_follow_the_softmax():
    l = np.array([0.0, 1.0, -1.0, 2.0, 0.5, -3.0])
    p = np.exp(l - sps.logsumexp(l))
    counts = np.zeros(l.size)
    for step in range(6000):
        g = oracle.gumbel(oracle.uniforms(21, step, 0, 0, oracle.STREAM_DRAFT, np.arange(l.size)))
        x, lp, gap, z = oracle.sample_decode(l, g)
        counts[x] += 1
        assert lp == pytest.approx(l[x] - sps.logsumexp(l)) and z == pytest.approx(sps.logsumexp(l))
        assert gap >= 0
    assert _chi2_p(counts, p) > 1e-3


def test_speculative_sampling_is_lossless():
    """The first token the block emits (x_0 if accepted, else the residual draw)
    is distributed as the target's p_0, whatever the draft's q_0; x_0 is
    accepted with probability sum_v min(p, q)."""
    ql = np.array([1.5, 0.0, -0.5, 0.7, -2.0])
    pl = np.array([0.2, 0.9, -0.3, -1.0, 0.4])
    pn = np.zeros(5)
    p = np.exp(pl - sps.logsumexp(pl))
    q = np.exp(ql - sps.logsumexp(ql))
    first = np.zeros(5)
    accepted = 0
    steps = 6000
    for step in range(steps):
        g = oracle.gumbel(oracle.uniforms(33, step, 0, 0, oracle.STREAM_DRAFT, np.arange(5)))
        x0 = int(np.argmax(ql + g))
        acc, bonus, info = oracle.verify_sampled([[x0]], ql[None, None, :], np.stack([pl, pn])[None], 33, step)
        if acc[0] == 1:
            accepted += 1
            first[x0] += 1
        else:
            first[bonus[0]] += 1
    assert _chi2_p(first, p) > 1e-3
    rate = np.minimum(p, q).sum()
    assert abs(accepted / steps - rate) < 4 * np.sqrt(rate * (1 - rate) / steps)


def test_speculative_sampling_special_cases():
    V = 7
    rng = np.random.default_rng(2)
    ql = rng.normal(size=(1, 3, V))
    # the target equals the draft: every token is accepted, the bonus comes from p_n
    T = np.concatenate([ql, rng.normal(size=(1, 1, V))], axis=1)
    for step in range(50):
        d = [[int(np.argmax(ql[0, j] + oracle.gumbel(oracle.uniforms(4, step, 0, j, 0, np.arange(V)))))
              for j in range(3)]]
        acc, bonus, _ = oracle.verify_sampled(d, ql, T, 4, step)
        key = T[0, 3] + oracle.gumbel(oracle.uniforms(4, step, 0, 3, oracle.STREAM_RESIDUAL, np.arange(V)))
        assert acc[0] == 3 and bonus[0] == int(np.argmax(key))
    # a draft token the target rules out (p = 0) is always rejected, and the
    # residual never gives it back
    T2 = T.copy()
    T2[0, 0, 2] = -np.inf
    for step in range(50):
        acc, bonus, _ = oracle.verify_sampled([[2, 0, 0]], ql, T2, 5, step)
        assert acc[0] == 0 and bonus[0] != 2


def test_draft_block_temperature_one_draws_with_the_drafting_stream():
    """Temperature 1: every position is argmax(l + g) of the same fused row as
    temperature 0, g the drafting-stream variates of (b, j); with a huge gap
    it agrees with the greedy draft."""
    base = synth.WORKLOADS["tiny"]
    w = synth.with_sizes(base, B=2, n=5)
    d = synth.make_inputs(w)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = oracle.log_prior(d["counts"])
    head = oracle.make_head(w.head, W)
    res = oracle.draft_block(head, d["long"], prior, 0.5, 0.5, sample=(9, 1), keep_fused=True)
    L = oracle.to_f64(d["long"])
    for b in range(2):
        for j in range(5):
            f = res.fused[b, j]
            if j == 0:
                np.testing.assert_array_equal(f, L[b, 0])
            g = oracle.gumbel(oracle.uniforms(9, 1, b, j, oracle.STREAM_DRAFT, np.arange(w.V)))
            assert res.tokens[b, j] == int(np.argmax(f + g))
            assert res.lse[b, j] == pytest.approx(sps.logsumexp(f))
            assert res.logp[b, j] == pytest.approx(f[res.tokens[b, j]] - sps.logsumexp(f))
    # the same run forced onto its own tokens reproduces them
    forced = oracle.draft_block(head, d["long"], prior, 0.5, 0.5, forced=res.tokens, sample=(9, 1))
    np.testing.assert_array_equal(forced.argmax, res.tokens)
    # scaled-up logits: the Gumbel noise cannot move the argmax
    big = oracle.draft_block(head, L * 1e4, prior, 0.0, 0.0, sample=(9, 1))
    greedy = oracle.draft_block(head, L * 1e4, prior, 0.0, 0.0)
    np.testing.assert_array_equal(big.tokens, greedy.tokens)
