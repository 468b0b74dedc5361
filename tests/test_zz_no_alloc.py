"""dels_combine_argmax_noalloc: the combine for callers that cannot allocate.

Some callers own only their input and output buffers (a plugin inside a host
framework whose allocator it cannot reach, or a loop where an allocation
could stall the device). This entry point serves them from a fixed scratch
compiled into the library. The test calls it through the C ABI twice in a
row on different inputs and compares it with dels_combine_argmax, which uses
a caller-provided workspace, within the combine tolerance of the parity
suite; it also checks that an oversized problem is rejected. Collected last
so that a failure here comes after every other test has run.
"""
import numpy as np
import pytest
import torch

import synth
import paper_2607_07409_gb300 as dels
from parity import LP_TOL_COMBINE

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _with_workspace(long, short, prior, w):
    rows, V = long.shape
    dt = dels.dtype_code(long)
    nbytes = dels.dels_combine_workspace_bytes(rows, V, dt)
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=DEV)
    out = [torch.empty(rows, dtype=torch.int32, device=DEV), torch.empty(rows, device=DEV),
           torch.empty(rows, device=DEV)]
    assert dels.dels_combine_argmax(long, short, dt, prior, w, w, rows, V, *out, ws, nbytes) == 0
    return out


def _no_alloc(long, short, prior, w):
    rows, V = long.shape
    out = [torch.full((rows,), -5, dtype=torch.int32, device=DEV), torch.empty(rows, device=DEV),
           torch.empty(rows, device=DEV)]
    r = dels.dels_combine_argmax_noalloc(long, short, dels.dtype_code(long), prior, w, w, rows, V, *out)
    assert r == 0, dels.dels_status_string(r)
    return out


def test_no_alloc_combine_matches_workspace_combine_twice():
    cases = [(7, 151936, "bf16", 0.5, 21), (300, 32000, "f32", 1.0, 22)]   # two calls in a row
    results = []
    for rows, V, dtype, w, seed in cases:
        d = synth.make_combine_inputs(rows, V, dtype, seed=seed, device=DEV)
        prior = dels.dels_prior_from_counts(d["counts"]).to(DEV)
        results.append((_no_alloc(d["long"], d["short"], prior, w), _with_workspace(d["long"], d["short"], prior, w)))
    torch.cuda.synchronize()
    for got, ref in results:
        np.testing.assert_array_equal(got[0].cpu().numpy(), ref[0].cpu().numpy())
        assert np.abs(got[1].cpu().numpy() - ref[1].cpu().numpy()).max() <= LP_TOL_COMBINE
        assert np.abs(got[2].cpu().numpy() - ref[2].cpu().numpy()).max() <= 2 * LP_TOL_COMBINE


def test_no_alloc_combine_many_rows_and_a_non_finite_row():
    """The four-rows-per-CTA plan (rows >= 64 x SMs), where the cleared ticket
    region has its largest size, and a row holding a NaN: the workspace status
    word is not readable here, so the row must come back as token -1 with a
    NaN log-probability while every other row matches the workspace combine."""
    rows, V = 20000, 64
    d = synth.make_combine_inputs(rows, V, "f32", seed=23, device=DEV)
    long = d["long"].clone()
    long[777, 5] = float("nan")
    prior = dels.dels_prior_from_counts(d["counts"]).to(DEV)
    got = _no_alloc(long, d["short"], prior, 0.5)
    ref = _with_workspace(long, d["short"], prior, 0.5)
    torch.cuda.synchronize()
    tok, lp = got[0].cpu().numpy(), got[1].cpu().numpy()
    assert tok[777] == -1 and np.isnan(lp[777])
    np.testing.assert_array_equal(tok, ref[0].cpu().numpy())
    keep = np.arange(rows) != 777
    assert np.abs(lp[keep] - ref[1].cpu().numpy()[keep]).max() <= LP_TOL_COMBINE
    assert ((tok[keep] >= 0) & (tok[keep] < V)).all()


def test_no_alloc_combine_rejects_bad_pointers_before_touching_its_scratch():
    """A rejected call enqueues nothing: a misaligned input is refused before
    the scratch is cleared, and the next call still matches the workspace path."""
    rows, V = 9, 4096
    d = synth.make_combine_inputs(rows, V, "bf16", seed=24, device=DEV)
    prior = dels.dels_prior_from_counts(d["counts"]).to(DEV)
    flat = d["long"].reshape(-1)
    out = [torch.empty(rows, dtype=torch.int32, device=DEV), torch.empty(rows, device=DEV), None]
    r = dels.dels_combine_argmax_noalloc(flat[1:], d["short"], dels.dtype_code(flat), prior, 0.5, 0.5, rows, V - 1,
                                         *out)
    assert r == dels.DELS_ERR_ALIGNMENT
    r = dels.dels_combine_argmax_noalloc(d["long"], d["short"], dels.dtype_code(flat), prior, 0.5, 0.5, rows, V,
                                         None, None, None)
    assert r == dels.DELS_ERR_NULL_POINTER
    got = _no_alloc(d["long"], d["short"], prior, 0.5)
    ref = _with_workspace(d["long"], d["short"], prior, 0.5)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(got[0].cpu().numpy(), ref[0].cpu().numpy())


def test_no_alloc_combine_rejects_problems_beyond_its_scratch():
    rows, V = 300000, 64
    big = torch.zeros(1, device=DEV)          # never read: the call must refuse before launching
    r = dels.dels_combine_argmax_noalloc(big, None, dels.DELS_F32, None, 0.0, 0.0, rows, V, big, None, None)
    assert r == dels.DELS_ERR_TOO_LARGE
