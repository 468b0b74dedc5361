"""GPU parity of temperature-1 drafting (Algorithm 1 with Decode = a draw from
the softmax by the Gumbel-max rule) against the oracle.

Both sides draw the same Philox4x32-10 uniforms, so a device token must be
the oracle's argmax of the keys l + g at every position, except where the
oracle's top-2 key gap is a near-tie (then within the tie tolerance of the
maximum key); the drafted prefix is re-checked in the oracle's forced mode.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
import paper_2607_07409_gb300 as dels
from parity import LP_TOL_BF16, LP_TOL_F32, check_draft, record
from test_gpu_parity import DEV, SMALL, _oracle_head, _with_table, _learned_weights

pytestmark = pytest.mark.gpu


def _sampled(name, seed=17, step=3, weights="learned"):
    w = synth.stress(SMALL[name])
    d = synth.make_inputs(w, device=DEV, target=False)
    if name == "gru_b64":
        d = _with_table(w, d)
    a, b = _learned_weights(w.n) if weights == "learned" else ([w.weight] * w.n, [w.weight] * w.n)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = dels.dels_prior_from_counts(d["counts"]).to(DEV)
    dr = dels.Drafter(w.head, W, w.B, w.n, w.V)
    tok, lp, gap, state = dr.sample(d["long"], prior, a, b, seed, step)
    torch.cuda.synchronize()
    assert dr.status() == 0
    W = {k: v for k, v in W.items() if k != "input_table"}
    return w, d, W, a, b, tok.cpu().numpy(), lp.cpu().numpy(), gap.cpu().numpy(), state


@pytest.mark.parametrize("name,seed,step", [("gru", 17, 3), ("gru_b64", 17, 3), ("gru_b100", 17, 3), ("mlp2", 17, 3),
                                            ("xfmr", 17, 3),
                                            ("markov", 17, 3), ("gru_f32", 17, 3), ("tiny", 17, 3),
                                            ("gru", 0xFEDCBA9876543210, 2 ** 32 - 1)])
def test_sampled_draft_matches_oracle(name, seed, step):
    """Every head; the last case puts both halves of the key and the whole
    step word of the counter to use."""
    w, d, W, a, b, tok, lp, gap, state = _sampled(name, seed, step)
    tol = LP_TOL_F32 if w.head.wdtype == "f32" else LP_TOL_BF16
    info = check_draft(tok, lp, gap, _oracle_head(w, W), d["long"].cpu(), oracle.log_prior(d["counts"]),
                       np.array(a), np.array(b), tol, sample=(seed, step))
    # the LSE of every fused row, kept for the verification
    lse = state[: w.B * w.n * 4].view(torch.float32).view(w.B, w.n).cpu().numpy()
    np.testing.assert_allclose(lse, info["ref"].lse, rtol=0, atol=tol * 4)
    print(name, record(f"sampled draft {name}", info))


def test_sampled_calls_reject_a_step_outside_the_counter_word():
    w = synth.stress(SMALL["gru"])
    d = synth.make_inputs(w, device=DEV, target=False)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = dels.dels_prior_from_counts(d["counts"]).to(DEV)
    dr = dels.Drafter(w.head, W, w.B, w.n, w.V)
    with pytest.raises(dels.DelsError) as e:
        dr.sample(d["long"], prior, [0.3] * w.n, [0.3] * w.n, 1, 2 ** 32)
    assert e.value.code == dels.DELS_ERR_BAD_SHAPE


def test_sampled_draft_depends_on_seed_and_step_only():
    w, d, W, a, b, tok1, lp1, _, _ = _sampled("gru", 5, 9)
    _, _, _, _, _, tok2, lp2, _, _ = _sampled("gru", 5, 9)
    np.testing.assert_array_equal(tok1, tok2)
    np.testing.assert_array_equal(lp1, lp2)
    _, _, _, _, _, tok3, _, _, _ = _sampled("gru", 5, 10)
    _, _, _, _, _, tok4, _, _, _ = _sampled("gru", 6, 9)
    assert not np.array_equal(tok1, tok3) and not np.array_equal(tok1, tok4)


def test_sampled_draft_first_token_frequencies_follow_the_softmax():
    """x_0 over many steps: empirical frequencies against softmax(l_L^(0)) of a
    small, flat row (every token has mass)."""
    from scipy.stats import chisquare
    V, B = 16, 64
    w = synth.Workload("flat", B=B, n=1, V=V, logit_dtype="f32",
                       head=synth.HeadSpec("markov", "f32", 0, 0, 16), weight=0.0, seed=3)
    d = synth.make_inputs(w, device=DEV, target=False)
    row = torch.linspace(-1.0, 1.0, V, device=DEV)
    long = row.expand(B, 1, V).contiguous()
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    dr = dels.Drafter(w.head, W, B, 1, V)
    prior = torch.zeros(V, device=DEV)
    counts = np.zeros(V)
    for step in range(40):
        tok, _, _, _ = dr.sample(long, prior, [0.0], [0.0], 99, step)
        counts += np.bincount(tok.cpu().numpy().ravel(), minlength=V)
    p = torch.softmax(row.double(), 0).cpu().numpy()
    assert chisquare(counts, counts.sum() * p).pvalue > 1e-3


# ------------------------------------------------ speculative-sampling verification

def _verify(w, d, W, a, b, tok, lp, state, target, seed, step):
    head = dels.make_head(w.head, W)
    tdt = dels.dtype_code(target)
    nbytes = dels.dels_verify_sampled_workspace_bytes(head, w.B, w.n, w.V, tdt)
    assert nbytes > 0
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=DEV)
    acc = torch.full((w.B,), -5, dtype=torch.int32, device=DEV)
    bonus = torch.full((w.B,), -5, dtype=torch.int32, device=DEV)
    bgap = torch.empty(w.B, dtype=torch.float32, device=DEV)
    prior = dels.dels_prior_from_counts(d["counts"]).to(DEV)
    r = dels.dels_verify_block_sampled(head, torch.as_tensor(tok, device=DEV), torch.as_tensor(lp, device=DEV), state,
                                       d["long"], dels.dtype_code(d["long"]), prior, a, b, target, tdt, w.B, w.n, w.V,
                                       seed, step, acc, bonus, bgap, ws, nbytes)
    assert r == 0, dels.dels_status_string(r)
    torch.cuda.synchronize()
    assert dels.dels_read_status(ws) == 0
    return acc.cpu().numpy(), bonus.cpu().numpy(), bgap.cpu().numpy()


def _check_verify(w, d, W, a, b, tok, acc, bonus, bgap, target, seed, step, lp_tol):
    """Accepted lengths and bonus tokens against the oracle run on the device's
    drafted tokens (the oracle rebuilds q from its own fused rows)."""
    ref = oracle.draft_block(_oracle_head(w, W), d["long"].cpu(), oracle.log_prior(d["counts"]), np.array(a),
                             np.array(b), forced=tok, sample=(seed, step), keep_fused=True)
    r_acc, r_bonus, info = oracle.verify_sampled(tok, ref.fused, target.cpu(), seed, step)
    # a test whose ratio p/q lies within the logprob tolerance of its uniform may go either way
    close = info["margin"] < 8 * lp_tol
    same_acc = acc == r_acc
    assert np.all(same_acc | close), (acc, r_acc, info["margin"])
    ok = same_acc & ~close
    # the bonus draw: identical unless the oracle's key gap is a near-tie
    tie = info["bonus_gap"] < 0.05
    bad = ok & (bonus != r_bonus) & ~tie
    assert not bad.any(), (bonus[bad], r_bonus[bad], info["bonus_gap"][bad])
    fin = ok & (bonus == r_bonus) & np.isfinite(info["bonus_gap"])
    return dict(requests=int(len(acc)), close=int(close.sum()), ties=int((ok & tie).sum()),
                accept=acc.tolist(), gap_err=float(np.abs(bgap[fin] - info["bonus_gap"][fin]).max(initial=0)))


@pytest.mark.parametrize("name", ["gru", "gru_b64", "mlp2", "xfmr", "markov", "gru_f32", "tiny"])
def test_sampled_verify_matches_oracle(name):
    seed, step = 23, 7
    w, d, W, a, b, tok, lp, gap, state = _sampled(name, seed, step)
    target = synth.make_target_logits(w, d["long"], device=DEV)
    acc, bonus, bgap = _verify(w, d, W, a, b, tok, lp, state, target, seed, step)
    tol = LP_TOL_F32 if w.head.wdtype == "f32" else LP_TOL_BF16
    info = _check_verify(w, d, W, a, b, tok, acc, bonus, bgap, target, seed, step, tol)
    print(name, info)
    assert np.all((acc >= 0) & (acc <= w.n)) and np.all((bonus >= 0) & (bonus < w.V))


@pytest.mark.parametrize("name", ["gru", "markov", "tiny"])
def test_sampled_verify_rejection_at_position_zero(name):
    """The target rules out every x_0 (p_0(x_0) = 0): every request rejects at
    0 and its bonus comes from the residual of softmax(l_L^(0)), never x_0."""
    seed, step = 31, 2
    w, d, W, a, b, tok, lp, gap, state = _sampled(name, seed, step)
    target = synth.make_target_logits(w, d["long"], device=DEV).clone()
    for bb in range(w.B):
        target[bb, 0, int(tok[bb, 0])] = float("-inf")
    acc, bonus, bgap = _verify(w, d, W, a, b, tok, lp, state, target, seed, step)
    assert np.all(acc == 0) and np.all(bonus != tok[:, 0])
    tol = LP_TOL_F32 if w.head.wdtype == "f32" else LP_TOL_BF16
    print(name, _check_verify(w, d, W, a, b, tok, acc, bonus, bgap, target, seed, step, tol))


def test_gumbel_transform_error_over_every_uniform():
    """The device's g = -ln(-ln u) for every one of the 2^23 uniforms a Philox
    word can give (u = (2k + 1) 2^-24), against the float64 transform: the
    largest absolute error stays below 4e-6 (the exponential variate E = -ln u
    carries a relative error of ~1.5e-6 at most, which g inherits as an
    absolute error, plus the fast outer logarithm's)."""
    k = torch.arange(1 << 23, dtype=torch.int64)
    w = k << 9                                   # the word's top 23 bits select k
    bits = torch.where(w >= 2 ** 31, w - 2 ** 32, w).to(torch.int32).to(DEV)   # same 32 bits, as int32
    g = torch.empty(1 << 23, dtype=torch.float32, device=DEV)
    assert dels.dels_selftest_gumbel(bits, g, 1 << 23) == 0
    torch.cuda.synchronize()
    u = (2.0 * np.arange(1 << 23, dtype=np.float64) + 1.0) / 2.0 ** 24
    exact = -np.log(-np.log(u))
    err = np.abs(g.cpu().numpy().astype(np.float64) - exact)
    worst = int(np.argmax(err))
    print(f"gumbel transform: max |error| {err[worst]:.3g} at u = {u[worst]:.9f}, mean {err.mean():.3g}")
    assert err[worst] < 4e-6
    assert dels.dels_selftest_gumbel(bits, g, -1) == dels.DELS_ERR_BAD_SHAPE
    assert dels.dels_selftest_gumbel(None, g, 1) == dels.DELS_ERR_NULL_POINTER
