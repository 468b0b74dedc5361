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


def test_no_alloc_combine_rejects_problems_beyond_its_scratch():
    rows, V = 300000, 64
    big = torch.zeros(1, device=DEV)          # never read: the call must refuse before launching
    r = dels.dels_combine_argmax_noalloc(big, None, dels.DELS_F32, None, 0.0, 0.0, rows, V, big, None, None)
    assert r == dels.DELS_ERR_TOO_LARGE
