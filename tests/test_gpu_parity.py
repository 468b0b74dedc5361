"""GPU parity of the C-ABI library against the CPU oracle.

Every call goes through libdels.so (via the ctypes binding); inputs are the
seeded synthetic workloads of ``synth``; expected values come from ``oracle``
only. Sizes are chosen so the oracle finishes in seconds while the device
path still runs several tiles and a ragged tail.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
import paper_2607_07409_gb300 as dels
from parity import LP_TOL_BF16, LP_TOL_F32, check_draft, check_rows, record

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _ws(nbytes):
    assert nbytes > 0
    return torch.zeros(nbytes, dtype=torch.uint8, device=DEV)


def _status(ws):
    return dels.dels_read_status(ws)


def _prior_input(counts):
    """float32 log prior [V] from the oracle (an input the device and the oracle share)."""
    return torch.from_numpy(oracle.log_prior(counts).astype(np.float32))


# ------------------------------------------------------------------ combine

def _combine(long, short, prior, alpha, beta):
    rows, V = long.shape
    dt = dels.dtype_code(long)
    nbytes = dels.dels_combine_workspace_bytes(rows, V, dt)
    ws = _ws(nbytes)
    tok = torch.full((rows,), -7, dtype=torch.int32, device=DEV)
    lp = torch.empty(rows, dtype=torch.float32, device=DEV)
    gap = torch.empty(rows, dtype=torch.float32, device=DEV)
    r = dels.dels_combine_argmax(long, short, dt, prior, alpha, beta, rows, V, tok, lp, gap, ws, nbytes)
    assert r == 0, dels.dels_status_string(r)
    torch.cuda.synchronize()
    return tok.cpu().numpy(), lp.cpu().numpy(), gap.cpu().numpy(), _status(ws)


@pytest.mark.parametrize("rows,V,dtype,w", [
    (5, 1000, "bf16", 0.5),        # ragged tail, one chunk per row
    (3, 1003, "f32", 1.0),         # V not a multiple of the vector width: scalar path
    (7, 1001, "bf16", 0.5),
    (64, 32000, "bf16", 0.0),      # w = 0: plain argmax, exact ties included
    (2, 151936, "f32", 0.5),       # few rows: split over many CTAs + last-CTA merge
    (1, 151936, "bf16", 1.0),
    (33, 5000, "f32", 0.0),
    (3, 1004, "f32", 0.5),         # V = 4 mod 8: element-wise path
    (5, 16392, "bf16", 0.5),       # rows cut between many CTAs
    (40, 32000, "f32", 0.3),       # one wave of resident CTAs
    (150, 20000, "bf16", 1.0),     # about one row per CTA
    (1217, 16000, "bf16", 0.5),    # more rows than one wave: two rows per CTA, an odd last pair
    (400, 50000, "bf16", 0.5),     # one wave of whole rows, a third of the slots idle
    (200, 50000, "f32", 0.0),      # the same at two CTAs per SM, exact ties
    (1023, 40000, "bf16", 1.0),    # one wave of row pairs, an odd last pair
])
def test_combine_matches_oracle(rows, V, dtype, w):
    d = synth.make_combine_inputs(rows, V, dtype, seed=rows * 31 + V, device=DEV)
    # the log prior is an input of the combine: both sides get the same float32 values (the oracle's)
    prior_in = _prior_input(d["counts"])
    tok, lp, gap, st = _combine(d["long"], d["short"], prior_in.to(DEV), w, w)
    assert st == 0
    rt, rl, rg = oracle.combine_argmax(d["long"], d["short"], prior_in.numpy().astype(np.float64), w, w)
    fused = None
    if rows * V < 5e6:
        fused = oracle.fuse(oracle.to_f64(d["long"]), oracle.to_f64(d["short"]),
                            prior_in.numpy().astype(np.float64), w, w)
    check_rows(tok, lp, gap, rt, rl, rg, exact_ties=(w == 0.0), fused=fused)


def test_combine_many_rows_grouped_path():
    rows, V = 10000, 64                      # rows >= 64 * SMs: 4 rows per CTA
    d = synth.make_combine_inputs(rows, V, "bf16", seed=11, device=DEV)
    prior = _prior_input(d["counts"])
    tok, lp, gap, st = _combine(d["long"], d["short"], prior.to(DEV), 0.5, 0.5)
    assert st == 0
    rt, rl, rg = oracle.combine_argmax(d["long"], d["short"], prior.numpy().astype(np.float64), 0.5, 0.5)
    check_rows(tok, lp, gap, rt, rl, rg)


def test_combine_optional_terms_absent():
    d = synth.make_combine_inputs(4, 4096, "f32", seed=12, device=DEV)
    tok, lp, gap, st = _combine(d["long"], None, None, 0.7, 0.7)
    assert st == 0
    rt, rl, rg = oracle.combine_argmax(d["long"], None, None, 0.7, 0.7)
    check_rows(tok, lp, gap, rt, rl, rg, exact_ties=True)


@pytest.mark.parametrize("V", [2048, 32768])      # row kernel / streamed rows
def test_combine_masked_and_nonfinite_rows(V):
    long = torch.randn(4, V, device=DEV) * 3
    long[0, :100] = -float("inf")            # masked entries are allowed
    long[1, :] = -float("inf")               # all masked: error
    long[2, V - 77] = float("nan")           # NaN: error
    long[3, 5] = float("inf")                # +inf: error
    tok, lp, gap, st = _combine(long, None, None, 0.0, 0.0)
    assert st & dels.DELS_STATUS_NONFINITE
    rt, rl, rg = oracle.combine_argmax(long[:1], None, None, 0.0, 0.0)
    assert tok[0] == rt[0] and abs(lp[0] - rl[0]) < 1e-5
    assert tok[1] == -1 and tok[2] == -1 and tok[3] == -1


def test_combine_nonfinite_rows_among_many():
    """A NaN, an all-masked row and an infinite entry among 400 rows each give
    token -1 and the status flag; the other rows match the oracle."""
    rows, V = 400, 50000
    long = torch.randn(rows, V, device=DEV) * 3
    long[7, 1234] = float("nan")
    long[8, :] = -float("inf")
    long[300, V - 1] = float("inf")
    tok, lp, gap, st = _combine(long, None, None, 0.0, 0.0)
    assert st & dels.DELS_STATUS_NONFINITE
    assert tok[7] == -1 and tok[8] == -1 and tok[300] == -1
    keep = [r for r in range(rows) if r not in (7, 8, 300)]
    rt, rl, rg = oracle.combine_argmax(long[keep], None, None, 0.0, 0.0)
    check_rows(tok[keep], lp[keep], gap[keep], rt, rl, rg, exact_ties=True)


def test_combine_zero_rows_is_noop():
    ws = _ws(4096)
    r = dels.dels_combine_argmax(None, None, dels.DELS_F32, None, 0.0, 0.0, 0, 100, None, None, None, ws, 4096)
    assert r == 0


# ------------------------------------------------------------------- verify

def _verify(draft, target):
    B, n = draft.shape
    V = target.shape[-1]
    dt = dels.dtype_code(target)
    nbytes = dels.dels_verify_workspace_bytes(B, n, V, dt)
    ws = _ws(nbytes)
    acc = torch.full((B,), -9, dtype=torch.int32, device=DEV)
    bonus = torch.full((B,), -9, dtype=torch.int32, device=DEV)
    targ = torch.full((B, n + 1), -9, dtype=torch.int32, device=DEV)
    r = dels.dels_verify_block(draft, target, dt, B, n, V, acc, bonus, targ, ws, nbytes)
    assert r == 0, dels.dels_status_string(r)
    torch.cuda.synchronize()
    return acc.cpu().numpy(), bonus.cpu().numpy(), targ.cpu().numpy(), _status(ws), (ws, nbytes)


@pytest.mark.parametrize("B,n,V,dtype", [
    (9, 6, 50, "bf16"), (5, 16, 151936, "bf16"), (3, 8, 32000, "f32"), (17, 4, 1003, "f32"), (2, 32, 4099, "bf16"),
    (4, 3, 1004, "f32"), (1, 1, 16384, "bf16"), (64, 16, 151936, "f32"),
])
def test_verify_planted_prefix(B, n, V, dtype):
    t, draft, planted, accept = synth.make_planted_verify(B, n, V, dtype, seed=B * n, device=DEV)
    acc, bonus, targ, st, _ = _verify(draft, t)
    assert st == 0
    np.testing.assert_array_equal(targ, planted.numpy())
    np.testing.assert_array_equal(acc, accept.numpy())
    np.testing.assert_array_equal(bonus, planted.numpy()[np.arange(B), accept.numpy()])


@pytest.mark.parametrize("B,n,V,dtype", [(40, 5, 3000, "bf16"), (6, 5, 32000, "bf16"), (5, 3, 20000, "f32")])
def test_verify_random_ties_match_oracle(B, n, V, dtype):
    """Small integer logits: many exact ties inside every quad, CTA and row,
    all resolved to the lowest index (row kernel and streamed rows)."""
    g = torch.Generator().manual_seed(3 + V)
    T = torch.randint(-3, 3, (B, n + 1, V), generator=g).to(torch.bfloat16 if dtype == "bf16" else torch.float32)
    draft = torch.randint(0, 2, (B, n), generator=g).to(torch.int32)
    acc, bonus, targ, st, _ = _verify(draft.to(DEV), T.to(DEV))
    ra, rb, rt = oracle.verify_greedy(draft.numpy(), T)
    np.testing.assert_array_equal(targ, rt)
    np.testing.assert_array_equal(acc, ra)
    np.testing.assert_array_equal(bonus, rb)


@pytest.mark.parametrize("V", [999, 40000])
def test_verify_repeated_calls_reuse_workspace(V):
    t, draft, planted, accept = synth.make_planted_verify(6, 7, V, "f32", seed=5, device=DEV)
    acc, bonus, targ, st, (ws, nbytes) = _verify(draft, t)
    for _ in range(3):   # tickets must reset between calls
        a2 = torch.empty(6, dtype=torch.int32, device=DEV)
        b2 = torch.empty(6, dtype=torch.int32, device=DEV)
        assert dels.dels_verify_block(draft, t, dels.DELS_F32, 6, 7, V, a2, b2, None, ws, nbytes) == 0
        torch.cuda.synchronize()
        np.testing.assert_array_equal(a2.cpu().numpy(), accept.numpy())


@pytest.mark.parametrize("V", [100, 16384])
def test_verify_bad_draft_token_flags_status(V):
    t, draft, planted, accept = synth.make_planted_verify(3, 4, V, "f32", seed=6, device=DEV)
    draft[2, 3] = V
    _, _, _, st, _ = _verify(draft, t)
    assert st & dels.DELS_STATUS_BAD_TOKEN


# ------------------------------------------------------------------ drafting

def _draft(w, d):
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = dels.dels_prior_from_counts(d["counts"]).to(DEV)
    drafter = dels.Drafter(w.head, W, w.B, w.n, w.V)
    tok, lp, gap = drafter(d["long"], prior, w.alpha, w.beta)
    torch.cuda.synchronize()
    assert drafter.status() == 0
    # the oracle takes its own prior from the same counts
    return tok.cpu().numpy(), lp.cpu().numpy(), gap.cpu().numpy(), W, oracle.log_prior(d["counts"])


def _oracle_head(w, W):
    return oracle.make_head(w.head, {k: v.cpu() for k, v in W.items()})


SMALL = {
    "tiny": synth.WORKLOADS["tiny"],
    "gru": synth.with_sizes(synth.WORKLOADS["qwen3_8b_batched"], B=5, n=6, V=3000,
                            head_d_model=256, head_d_hidden=128, head_d_rank=64),
    "gru_b64": synth.with_sizes(synth.WORKLOADS["qwen3_8b_batched"], B=64, n=4, V=4096,
                                head_d_model=512, head_d_hidden=256, head_d_rank=256),
    # more than 64 requests: one 128-row copy of the activations, all four TMEM lane quadrants live
    "gru_b100": synth.with_sizes(synth.WORKLOADS["qwen3_8b_batched"], B=100, n=3, V=2048,
                                 head_d_model=256, head_d_hidden=128, head_d_rank=128),
    "mlp2": synth.with_sizes(synth.WORKLOADS["qwen3_0p6b"], B=3, n=6, V=2000,
                             head_d_model=128, head_d_hidden=192, head_d_rank=192),
    # more requests than the CUDA-core path takes: tensor-core products + reductions
    "mlp2_b9": synth.with_sizes(synth.WORKLOADS["qwen3_0p6b"], B=9, n=5, V=2000,
                                head_d_model=128, head_d_hidden=192, head_d_rank=192),
    "xfmr": synth.with_sizes(synth.WORKLOADS["qwen3_4b"], B=2, n=5, V=1536,
                             head_d_model=256, head_d_hidden=512, head_d_rank=256, head_n_heads=4,
                             head_max_pos=8),
    # 3B = 144 three-term rows: the head's products run as two row blocks (128 + 16)
    "xfmr_b48": synth.with_sizes(synth.WORKLOADS["qwen3_4b"], B=48, n=4, V=1024,
                                 head_d_model=128, head_d_hidden=256, head_d_rank=128, head_n_heads=4,
                                 head_max_pos=4),
    "markov": synth.Workload("markov", B=4, n=6, V=2048, logit_dtype="bf16",
                             head=synth.HeadSpec("markov", "bf16", 0, 0, 128), weight=0.5, seed=7),
    "markov_f32": synth.Workload("markov_f32", B=2, n=5, V=1000, logit_dtype="f32",
                                 head=synth.HeadSpec("markov", "f32", 0, 0, 64), weight=0.5, seed=8),
    # the wide vocabulary projection: a 4096-wide state (no recurrence), K = 4096 streamed with W
    "markov_wide": synth.Workload("markov_wide", B=40, n=4, V=1536, logit_dtype="bf16",
                                  head=synth.HeadSpec("markov", "bf16", 0, 0, 4096), weight=0.5, seed=9),
    "gru_f32": synth.with_sizes(synth.WORKLOADS["qwen3_8b_batched"], B=3, n=5, V=1200, logit_dtype="f32",
                                head_wdtype="f32", head_d_model=64, head_d_hidden=32, head_d_rank=16),
}


@pytest.mark.parametrize("stress", [False, True])
@pytest.mark.parametrize("name", list(SMALL))
def test_draft_small_matches_oracle(name, stress):
    w = SMALL[name]
    if stress:
        w = synth.stress(w)
    d = synth.make_inputs(w, device=DEV, target=False)
    tok, lp, gap, W, prior = _draft(w, d)
    tol = LP_TOL_F32 if w.head.wdtype == "f32" else LP_TOL_BF16
    info = check_draft(tok, lp, gap, _oracle_head(w, W), d["long"].cpu(), prior, w.alpha, w.beta, tol)
    print(name, stress, record(f"draft {name}, stress {stress}", info))


@pytest.mark.parametrize("stress", [False, True])
@pytest.mark.parametrize("name", ["gru", "gru_b64"])
def test_draft_persistent_kernel_matches_oracle(name, stress, monkeypatch):
    # the one-launch-per-block drafting path for bf16 GRU heads
    monkeypatch.setenv("DELS_DRAFT_PERSISTENT", "1")
    w = SMALL[name]
    if stress:
        w = synth.stress(w)
    d = synth.make_inputs(w, device=DEV, target=False)
    tok, lp, gap, W, prior = _draft(w, d)
    info = check_draft(tok, lp, gap, _oracle_head(w, W), d["long"].cpu(), prior, w.alpha, w.beta, LP_TOL_BF16)
    print(name, stress, info)


def _with_table(w, d):
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    d = dict(d)
    d["head.input_table"] = dels.gru_input_table(w.head, W, w.V)
    return d


@pytest.mark.parametrize("V", [3000, 4096])
def test_gru_input_table_is_the_input_product(V):
    w = synth.with_sizes(synth.stress(synth.WORKLOADS["qwen3_8b_batched"]), B=2, n=2, V=V,
                         head_d_model=256, head_d_hidden=128, head_d_rank=64)
    d = synth.make_inputs(w, device=DEV, target=False)
    G = _with_table(w, d)["head.input_table"]
    torch.cuda.synchronize()
    E = d["head.emb"].double().cpu()
    Wih = d["head.w_ih"].double().cpu()
    ref = E @ Wih.T
    got = G.double().cpu()
    assert got.shape == ref.shape
    # bf16 x bf16 products are exact in f32; only the f32 summation of d_model
    # terms rounds: |error| <= d_model * 2^-23 * sum |E_k W_k| (standard bound)
    bound = w.head.d_model * 2.0 ** -23 * (E.abs() @ Wih.abs().T) + 1e-30
    assert torch.all((got - ref).abs() <= bound), float(((got - ref).abs() / bound).max())


@pytest.mark.parametrize("stress", [False, True])
@pytest.mark.parametrize("name", ["gru", "gru_b64"])
def test_draft_with_input_table_matches_oracle(name, stress):
    w = SMALL[name]
    if stress:
        w = synth.stress(w)
    d = _with_table(w, synth.make_inputs(w, device=DEV, target=False))
    tok, lp, gap, W, prior = _draft(w, d)
    W = {k: v for k, v in W.items() if k != "input_table"}
    info = check_draft(tok, lp, gap, _oracle_head(w, W), d["long"].cpu(), prior, w.alpha, w.beta, LP_TOL_BF16)
    # the fused merge's ticket resets itself: a second call gives the same block
    tok2, lp2, gap2, _, _ = _draft(w, d)
    np.testing.assert_array_equal(tok2, tok)
    np.testing.assert_array_equal(lp2, lp)
    print(name, stress, info)


@pytest.mark.parametrize("stress", [False, True])
@pytest.mark.parametrize("name", ["gru", "gru_b64"])
def test_draft_fused_products_vocab_kernel_matches_oracle(name, stress, monkeypatch):
    # the input-table path with the products and the vocabulary projection in one cooperative launch
    monkeypatch.setenv("DELS_DRAFT_FUSED", "1")
    w = SMALL[name]
    if stress:
        w = synth.stress(w)
    d = _with_table(w, synth.make_inputs(w, device=DEV, target=False))
    tok, lp, gap, W, prior = _draft(w, d)
    W = {k: v for k, v in W.items() if k != "input_table"}
    info = check_draft(tok, lp, gap, _oracle_head(w, W), d["long"].cpu(), prior, w.alpha, w.beta, LP_TOL_BF16)
    tok2, _, _, _, _ = _draft(w, d)
    np.testing.assert_array_equal(tok2, tok)
    print(name, stress, info)


def _learned_weights(n):
    """Per-position (alpha_j, beta_j) from the Appendix C table (positions 2..15
    are j = 1..14; later positions keep the last printed value)."""
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "appendix_c_learned_weights.txt")
    rows = [l.split() for l in open(path) if l.strip() and not l.startswith("#")]
    tab = {int(p): (float(a), float(b)) for p, a, b in rows}
    a, b = [0.0] * n, [0.0] * n
    for j in range(1, n):
        a[j], b[j] = tab[min(j + 1, max(tab))]
    return a, b


@pytest.mark.parametrize("name", ["gru", "gru_b64", "mlp2", "xfmr", "markov", "gru_f32", "tiny"])
def test_draft_per_position_weights_match_oracle(name):
    w = synth.stress(SMALL[name])
    d = synth.make_inputs(w, device=DEV, target=False)
    if name == "gru_b64":
        d = _with_table(w, d)
    a, b = _learned_weights(w.n)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = dels.dels_prior_from_counts(d["counts"]).to(DEV)
    dr = dels.Drafter(w.head, W, w.B, w.n, w.V)
    tok, lp, gap = dr(d["long"], prior, a, b)
    torch.cuda.synchronize()
    assert dr.status() == 0
    W = {k: v for k, v in W.items() if k != "input_table"}
    tol = LP_TOL_F32 if w.head.wdtype == "f32" else LP_TOL_BF16
    info = check_draft(tok.cpu().numpy(), lp.cpu().numpy(), gap.cpu().numpy(), _oracle_head(w, W), d["long"].cpu(),
                       oracle.log_prior(d["counts"]), np.array(a), np.array(b), tol)
    print(name, info)


def test_draft_zero_weight_is_dflash_argmax():
    w = synth.with_sizes(synth.stress(synth.WORKLOADS["qwen3_8b_batched"]), B=8, n=5, V=2048, weight=0.0,
                         head_d_model=128, head_d_hidden=64, head_d_rank=64)
    d = synth.make_inputs(w, device=DEV, target=False)
    tok, lp, gap, W, prior = _draft(w, d)
    L = oracle.to_f64(d["long"])
    np.testing.assert_array_equal(tok, np.argmax(L, axis=2))


def test_draft_block_of_one_position():
    w = synth.with_sizes(synth.WORKLOADS["qwen3_8b_batched"], B=3, n=1, V=1024,
                         head_d_model=64, head_d_hidden=32, head_d_rank=32)
    d = synth.make_inputs(w, device=DEV, target=False)
    tok, lp, gap, W, prior = _draft(w, d)
    L = oracle.to_f64(d["long"])
    np.testing.assert_array_equal(tok[:, 0], np.argmax(L[:, 0], axis=1))


@pytest.mark.parametrize("table", [False, True])
def test_draft_largest_batch_tile(table):
    """B = 128: every row of the tensor cores' M = 128 tile is a live request."""
    w = synth.with_sizes(synth.stress(synth.WORKLOADS["qwen3_8b_batched"]), B=128, n=4, V=2048,
                         head_d_model=128, head_d_hidden=64, head_d_rank=64)
    d = synth.make_inputs(w, device=DEV, target=False)
    if table:
        d = _with_table(w, d)
    tok, lp, gap, W, prior = _draft(w, d)
    W = {k: v for k, v in W.items() if k != "input_table"}
    print(check_draft(tok, lp, gap, _oracle_head(w, W), d["long"].cpu(), prior, w.alpha, w.beta, LP_TOL_BF16))


def test_draft_and_sampled_calls_with_an_empty_batch():
    w = synth.with_sizes(synth.WORKLOADS["qwen3_8b_batched"], B=2, n=4, V=1024,
                         head_d_model=64, head_d_hidden=32, head_d_rank=32)
    d = synth.make_inputs(w, device=DEV, target=True)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    head = dels.make_head(w.head, W)
    prior = dels.dels_prior_from_counts(d["counts"]).to(DEV)
    ws = _ws(dels.dels_draft_workspace_bytes(head, 2, w.n, w.V))
    nb = ws.numel()
    tok = torch.full((1,), -9, dtype=torch.int32, device=DEV)
    lp = torch.zeros(1, device=DEV)
    assert dels.dels_draft_block(head, d["long"], dels.DELS_BF16, prior, 0.3, 0.3, 0, w.n, w.V, tok, lp, None,
                                 ws, nb) == 0
    a = [0.3] * w.n
    st = _ws(max(16, dels.dels_draft_state_bytes(head, 1, w.n)))
    assert dels.dels_draft_block_sampled(head, d["long"], dels.DELS_BF16, prior, a, a, 0, w.n, w.V, 1, 2, tok, lp,
                                         None, st, st.numel(), ws, nb) == 0
    vb = dels.dels_verify_sampled_workspace_bytes(head, 1, w.n, w.V, dels.DELS_BF16)
    vws = _ws(vb)
    acc = torch.full((1,), -9, dtype=torch.int32, device=DEV)
    assert dels.dels_verify_block_sampled(head, tok, lp, st, d["long"], dels.DELS_BF16, prior, a, a, d["target"],
                                          dels.DELS_BF16, 0, w.n, w.V, 1, 2, acc, acc, None, vws, vb) == 0
    torch.cuda.synchronize()
    assert int(tok[0]) == -9 and int(acc[0]) == -9      # nothing was written
    assert _status(ws) == 0 and _status(vws) == 0


@pytest.mark.parametrize("table", [False, True])
def test_draft_nonfinite_long_logits_flag_the_row(table):
    """A NaN in request 1's DFlash logits at position 2: the status word flags
    it, that position's token is -1, and the other requests are untouched."""
    w = synth.with_sizes(synth.stress(synth.WORKLOADS["qwen3_8b_batched"]), B=4, n=5, V=2048,
                         head_d_model=128, head_d_hidden=64, head_d_rank=64)
    d = synth.make_inputs(w, device=DEV, target=False)
    if table:
        d = _with_table(w, d)
    d["long"][1, 2, 77] = float("nan")
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = dels.dels_prior_from_counts(d["counts"]).to(DEV)
    dr = dels.Drafter(w.head, W, w.B, w.n, w.V)
    tok, lp, gap = dr(d["long"], prior, w.alpha, w.beta)
    torch.cuda.synchronize()
    assert dr.status() & dels.DELS_STATUS_NONFINITE
    tok, lp, gap = tok.cpu().numpy(), lp.cpu().numpy(), gap.cpu().numpy()
    assert tok[1, 2] == -1 and np.isnan(lp[1, 2])
    rows = [0, 2, 3]
    W = {k: v for k, v in W.items() if k != "input_table"}
    check_draft(tok[rows], lp[rows], gap[rows], _oracle_head(w, W), d["long"][rows].cpu(),
                oracle.log_prior(d["counts"]), w.alpha, w.beta, LP_TOL_BF16)


# ------------------------------------------------------------ bounded waits

def test_expired_wait_reports_timeout_and_context_survives():
    nbytes = dels.dels_selftest_timeout_bytes()
    ws = _ws(nbytes)
    assert dels.dels_selftest_timeout(ws, nbytes) == 0
    st = _status(ws)
    assert st & dels.DELS_STATUS_TIMEOUT, st
    # the context is still usable: an ordinary call runs and is correct
    d = synth.make_combine_inputs(3, 4096, "bf16", seed=5, device=DEV)
    prior = _prior_input(d["counts"])
    tok, lp, gap, st2 = _combine(d["long"], d["short"], prior.to(DEV), 0.5, 0.5)
    assert st2 == 0
    rt, rl, rg = oracle.combine_argmax(d["long"], d["short"], prior.numpy().astype(np.float64), 0.5, 0.5)
    check_rows(tok, lp, gap, rt, rl, rg)
