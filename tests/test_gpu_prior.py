"""GPU parity of the device unigram-prior estimation (Appendix A) against the oracle.

Counts and tallies are integers and must match bit for bit. The log prior is
evaluated in float64 on both sides and stored as float32 by the device, so
each entry must lie within one float32 spacing of the oracle's fp64 value.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
import paper_2607_07409_gb300 as dels

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _ws(V, N):
    n = dels.dels_prior_workspace_bytes(V, N)
    assert n > 0
    return torch.zeros(n, dtype=torch.uint8, device=DEV), n


def _check_log_prior(got, counts, lam):
    ref = oracle.log_prior(counts, lam)
    ulp = np.spacing(np.abs(ref).astype(np.float32)).astype(np.float64)
    err = np.abs(got.cpu().numpy().astype(np.float64) - ref)
    assert np.all(err <= ulp), f"max error {err.max()} ulp {ulp[np.argmax(err)]}"


def _estimate(tok, mask, V, lam=1.0):
    out, counts, tally = dels.estimate_prior(tok, mask, V, lam)
    torch.cuda.synchronize()
    return out, counts.cpu().numpy(), tally.cpu().numpy()


def _corpus(V, N, seed, bad=0):
    tok, mask = synth.make_corpus(V, N, seed)
    if bad:
        g = torch.Generator().manual_seed(seed)
        where = torch.randperm(N, generator=g)[:bad]
        tok[where] = torch.tensor([-1, V, V + 7, -(2 ** 31)], dtype=torch.int32).repeat(bad)[:bad]
        mask[where] = 1
    return tok, mask


@pytest.mark.parametrize("V,N,seed,lam", [
    (1000, 100003, 1, 1.0),        # ragged tail after the vector range
    (151936, 1 << 20, 2, 1.0),
    (32000, 511, 3, 0.5),          # shorter than one warp step: all scalar
    (7, 4096, 4, 2.0),             # tiny vocabulary: every id hot
])
def test_estimate_matches_oracle(V, N, seed, lam):
    tok, mask = _corpus(V, N, seed)
    c_ref, n_in, n_out = oracle.count_masked_tokens(tok.numpy(), mask.numpy(), V)
    out, c, tally = _estimate(tok.to(DEV), mask.to(DEV), V, lam)
    np.testing.assert_array_equal(c, c_ref)
    assert tally.tolist() == [n_in, n_out]
    _check_log_prior(out, c_ref, lam)


def test_out_of_range_ids_are_tallied_and_flagged():
    V, N = 5000, 70001
    tok, mask = _corpus(V, N, 5, bad=37)
    c_ref, n_in, n_out = oracle.count_masked_tokens(tok.numpy(), mask.numpy(), V)
    assert n_out == 37
    ws, nbytes = _ws(V, N)
    out = torch.empty(V, dtype=torch.float32, device=DEV)
    counts = torch.empty(V, dtype=torch.int64, device=DEV)
    tally = torch.empty(2, dtype=torch.int64, device=DEV)
    r = dels.dels_prior_estimate(tok.to(DEV), mask.to(DEV), N, V, 1.0, out, counts, tally, ws, nbytes)
    assert r == 0
    assert dels.dels_read_status(ws) == dels.DELS_STATUS_BAD_TOKEN
    np.testing.assert_array_equal(counts.cpu().numpy(), c_ref)
    assert tally.cpu().tolist() == [n_in, n_out]
    _check_log_prior(out, c_ref, 1.0)


@pytest.mark.parametrize("tok_off,mask_off", [(1, 1), (2, 2), (3, 3), (1, 0), (0, 3), (2, 1)])
def test_unaligned_corpus_pieces(tok_off, mask_off):
    """Offsets into a larger corpus: equal offsets keep a vector range, others go one by one."""
    V, N = 3000, 40000
    tok, mask = _corpus(V, N + 8, 6)
    t_dev, m_dev = tok.to(DEV), mask.to(DEV)
    n = N - 5
    c_ref, n_in, n_out = oracle.count_masked_tokens(tok[tok_off:tok_off + n].numpy(),
                                                    mask[mask_off:mask_off + n].numpy(), V)
    ws, nbytes = _ws(V, n)
    counts = torch.zeros(V, dtype=torch.int64, device=DEV)
    tally = torch.zeros(2, dtype=torch.int64, device=DEV)
    r = dels.dels_prior_count(t_dev[tok_off:], m_dev[mask_off:], n, V, counts, tally, ws, nbytes)
    assert r == 0
    torch.cuda.synchronize()
    np.testing.assert_array_equal(counts.cpu().numpy(), c_ref)
    assert tally.cpu().tolist() == [n_in, n_out]


def test_pieces_accumulate_then_log_equals_one_call():
    V, N = 151936, 300000
    tok, mask = _corpus(V, N, 7)
    t_dev, m_dev = tok.to(DEV), mask.to(DEV)
    ws, nbytes = _ws(V, N)
    counts = torch.zeros(V, dtype=torch.int64, device=DEV)
    tally = torch.zeros(2, dtype=torch.int64, device=DEV)
    cuts = [0, 12345, 12346, 200000, N]
    for a, b in zip(cuts[:-1], cuts[1:]):
        assert dels.dels_prior_count(t_dev[a:], m_dev[a:], b - a, V, counts, tally, ws, nbytes) == 0
    out = torch.empty(V, dtype=torch.float32, device=DEV)
    assert dels.dels_prior_log(counts, V, 1.0, out, ws, nbytes) == 0
    c_ref, n_in, _ = oracle.count_masked_tokens(tok.numpy(), mask.numpy(), V)
    np.testing.assert_array_equal(counts.cpu().numpy(), c_ref)
    assert tally.cpu().tolist() == [n_in, 0]
    _check_log_prior(out, c_ref, 1.0)
    # the ticket of the two-level sum is re-armed: a second call gives the same result
    out2 = torch.empty_like(out)
    assert dels.dels_prior_log(counts, V, 1.0, out2, ws, nbytes) == 0
    assert torch.equal(out, out2)
    one, c1, _ = _estimate(t_dev, m_dev, V)
    assert torch.equal(one, out)


def test_empty_corpus_and_all_unmasked_give_the_uniform_prior():
    V = 1000
    ref = np.full(V, -np.log(V))
    for tok, mask in ((torch.zeros(0, dtype=torch.int32), torch.zeros(0, dtype=torch.uint8)),
                      (torch.arange(5000, dtype=torch.int32) % V, torch.zeros(5000, dtype=torch.uint8))):
        out, c, tally = _estimate(tok.to(DEV), mask.to(DEV), V)
        assert not c.any() and tally.tolist() == [0, 0]
        _check_log_prior(out, np.zeros(V, np.int64), 1.0)
        np.testing.assert_allclose(out.cpu().numpy(), ref, rtol=1e-7)


def test_single_hot_id_and_nonunit_mask_bytes():
    """Every position the same id (all atomics on one address) and mask bytes other than 1."""
    V, N = 151936, (1 << 22) + 3
    tok = torch.full((N,), 4242, dtype=torch.int32)
    mask = torch.full((N,), 255, dtype=torch.uint8)
    mask[::3] = 0
    out, c, tally = _estimate(tok.to(DEV), mask.to(DEV), V)
    expect = int((mask != 0).sum())
    assert c[4242] == expect and c.sum() == expect and tally.tolist() == [expect, 0]
    c_ref = np.zeros(V, np.int64)
    c_ref[4242] = expect
    _check_log_prior(out, c_ref, 1.0)


def test_full_corpus_counts_match_oracle():
    """The benchmark corpus: 2^28 positions over V = 151936, generated on the device."""
    w = synth.WORKLOADS["qwen3_8b_batched"]
    tok, mask = synth.make_corpus(w.V, synth.CORPUS_TOKENS, w.seed, device=DEV)
    out, c, tally = _estimate(tok, mask, w.V)
    c_ref, n_in, n_out = oracle.count_masked_tokens(tok.cpu().numpy(), mask.cpu().numpy(), w.V)
    np.testing.assert_array_equal(c, c_ref)
    assert tally.tolist() == [n_in, n_out]
    _check_log_prior(out, c_ref, 1.0)


# ------------------------------------------------------------- the hot/cold path
# (large vocabularies over long ranges: a prefix counted exactly, the most
# frequent ids so far on chip, the others through per-CTA cold buffers)

HOT_N = (1 << 24) + 1234


def test_hot_cold_path_matches_oracle_with_bad_ids():
    V = 151936
    tok, mask = _corpus(V, HOT_N, 8, bad=101)
    c_ref, n_in, n_out = oracle.count_masked_tokens(tok.numpy(), mask.numpy(), V)
    ws, nbytes = _ws(V, HOT_N)
    out = torch.empty(V, dtype=torch.float32, device=DEV)
    counts = torch.empty(V, dtype=torch.int64, device=DEV)
    tally = torch.empty(2, dtype=torch.int64, device=DEV)
    assert dels.dels_prior_estimate(tok.to(DEV), mask.to(DEV), HOT_N, V, 1.0, out, counts, tally, ws, nbytes) == 0
    assert dels.dels_read_status(ws) == dels.DELS_STATUS_BAD_TOKEN
    np.testing.assert_array_equal(counts.cpu().numpy(), c_ref)
    assert tally.cpu().tolist() == [n_in, n_out] and n_out == 101
    _check_log_prior(out, c_ref, 1.0)


def test_hot_cold_path_when_the_prefix_misleads():
    """The prefix holds one id only, the rest is uniform over V: almost every
    later position is cold and the cold buffers overflow into direct adds."""
    V = 151936
    g = torch.Generator().manual_seed(9)
    tok = torch.randint(0, V, (HOT_N,), generator=g, dtype=torch.int32)
    tok[: 1 << 23] = 77
    mask = (torch.rand(HOT_N, generator=g) < 0.9).to(torch.uint8)
    c_ref, n_in, n_out = oracle.count_masked_tokens(tok.numpy(), mask.numpy(), V)
    out, c, tally = _estimate(tok.to(DEV), mask.to(DEV), V)
    np.testing.assert_array_equal(c, c_ref)
    assert tally.tolist() == [n_in, n_out]


def test_hot_cold_pieces_on_top_of_earlier_counts():
    """A second long piece chooses its hot set from counts that already hold the first."""
    V = 151936
    tok, mask = _corpus(V, 2 * HOT_N, 10)
    t_dev, m_dev = tok.to(DEV), mask.to(DEV)
    ws, nbytes = _ws(V, HOT_N)
    counts = torch.zeros(V, dtype=torch.int64, device=DEV)
    tally = torch.zeros(2, dtype=torch.int64, device=DEV)
    for a in (0, HOT_N):
        assert dels.dels_prior_count(t_dev[a:], m_dev[a:], HOT_N, V, counts, tally, ws, nbytes) == 0
    torch.cuda.synchronize()
    c_ref, n_in, _ = oracle.count_masked_tokens(tok.numpy(), mask.numpy(), V)
    np.testing.assert_array_equal(counts.cpu().numpy(), c_ref)
    assert tally.cpu().tolist() == [n_in, 0]


def test_hot_path_hand_off_of_a_single_id():
    """One id at every loss-masked position of a hot-path range: every CTA's
    16-bit bin for it passes 2^15 twice and hands it to the global count."""
    V, N = 151936, HOT_N
    tok = torch.full((N,), 4242, dtype=torch.int32)
    mask = torch.full((N,), 3, dtype=torch.uint8)
    mask[::3] = 0
    out, c, tally = _estimate(tok.to(DEV), mask.to(DEV), V)
    expect = int((mask != 0).sum())
    assert expect // torch.cuda.get_device_properties(0).multi_processor_count > 2 * 2 ** 15
    assert c[4242] == expect and c.sum() == expect and tally.tolist() == [expect, 0]


def test_hot_path_vocabulary_a_multiple_of_15_with_bad_ids():
    """V = 15 * 10129: an id clamped to V falls on the remap table's zero
    sentinel word, past the last word that holds vocabulary ids."""
    V = 151935
    tok, mask = _corpus(V, HOT_N, 11, bad=57)
    c_ref, n_in, n_out = oracle.count_masked_tokens(tok.numpy(), mask.numpy(), V)
    out, c, tally = _estimate(tok.to(DEV), mask.to(DEV), V)
    np.testing.assert_array_equal(c, c_ref)
    assert tally.tolist() == [n_in, n_out] and n_out == 57
