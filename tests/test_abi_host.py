"""Host-side checks of the C-ABI library (no GPU needed).

The library must load, export every entry point ``include/dels.h`` declares,
and reject bad arguments on the host before touching a device.
"""
import ctypes
import os
import re

import numpy as np
import pytest
import torch

import oracle
import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def dels():
    import paper_2607_07409_gb300 as m
    if not os.path.exists(m.library_path()):
        from paper_2607_07409_gb300 import build
        build.build()
    m.lib()
    return m


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "dels.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dels_[a-z0-9_]+)\s*\(", src)))


def test_library_exports_every_declared_symbol(dels):
    declared = _declared_functions()
    assert len(declared) >= 10
    L = ctypes.CDLL(dels.library_path())
    for name in declared:
        assert hasattr(L, name), f"missing export {name}"
    assert sorted(dels.exported_symbols()) == declared


def test_binding_codes_match_the_header(dels):
    src = open(os.path.join(ROOT, "include", "dels.h")).read()
    codes = dict((k, int(v)) for k, v in re.findall(r"\b(DELS_(?:ERR|STATUS)_[A-Z_]+)\s*=\s*(-?\d+)", src))
    assert len(codes) >= 11
    for name, value in codes.items():
        assert getattr(dels, name) == value, name


def test_version_and_status_strings(dels):
    assert dels.dels_version() >= 100
    assert dels.dels_status_string(0) == "ok"
    assert "NaN" in dels.dels_status_string(1) or "non-finite" in dels.dels_status_string(1)
    assert dels.dels_status_string(-4).startswith("pointer")


def test_prior_from_counts_matches_oracle(dels):
    c = synth.make_counts(synth.WORKLOADS["qwen3_8b_batched"])
    got = dels.dels_prior_from_counts(c).numpy().astype(np.float64)
    ref = oracle.log_prior(c)
    np.testing.assert_allclose(got, ref, rtol=0, atol=2e-6)    # float32 storage of an fp64 value
    got2 = dels.dels_prior_from_counts(torch.tensor([0, 1, 2]), lam=0.5).numpy()
    np.testing.assert_allclose(got2, np.log(np.array([0.5, 1.5, 2.5]) / 4.5), atol=1e-7)


def test_prior_rejects_bad_arguments(dels):
    L = dels.lib()
    out = torch.empty(3)
    c = torch.tensor([1, -1, 2])
    assert L.dels_prior_from_counts(c.data_ptr(), 3, 1.0, out.data_ptr()) == -2
    c = torch.tensor([1, 1, 2])
    assert L.dels_prior_from_counts(c.data_ptr(), 3, 0.0, out.data_ptr()) == -2
    assert L.dels_prior_from_counts(None, 3, 1.0, out.data_ptr()) == -1


def test_host_validation_rejects_before_device_work(dels):
    L = dels.lib()
    ws = ctypes.create_string_buffer(1024)
    wsp = ctypes.addressof(ws)
    # unknown dtype code
    assert L.dels_combine_argmax(16, 16, 7, None, 0.0, 0.0, 1, 8, 16, None, None, wsp, 1024, None) == -3
    # negative rows
    assert L.dels_combine_argmax(16, 16, 0, None, 0.0, 0.0, -1, 8, 16, None, None, wsp, 1024, None) == -2
    # missing output
    assert L.dels_combine_argmax(16, None, 0, None, 0.0, 0.0, 1, 8, None, None, None, wsp, 1024, None) == -1
    # misaligned logits
    assert L.dels_combine_argmax(18, None, 0, None, 0.0, 0.0, 1, 8, 16, None, None, wsp, 1024, None) == -4
    # no workspace
    assert L.dels_combine_argmax(16, None, 0, None, 0.0, 0.0, 1, 8, 16, None, None, None, 0, None) == -5
    # verify: n out of range
    assert L.dels_verify_block(16, 16, 0, 1, 0, 8, 16, 16, None, wsp, 1024, None) == -2
    assert L.dels_verify_block(16, 16, 0, 1, 2000, 8, 16, 16, None, wsp, 1024, None) == -2
    # rows == 0 and B == 0 are no-ops
    assert L.dels_combine_argmax(None, None, 0, None, 0.0, 0.0, 0, 8, None, None, None, wsp, 1024, None) == 0
    assert L.dels_verify_block(None, None, 0, 0, 4, 8, None, None, None, wsp, 1024, None) == 0


def test_draft_validation(dels):
    L = dels.lib()
    spec = synth.WORKLOADS["qwen3_8b_batched"].head
    h = dels.LocalHead()
    h.kind, h.wdtype = 0, 1
    h.d_model, h.d_hidden, h.d_rank = spec.d_model, spec.d_hidden, spec.d_rank
    h.emb, h.w_vocab = 4096, 8192
    h.w[0], h.w[1], h.w[2] = 16, 32, 48
    ws = 64
    args = lambda B, n, V, dt=1: (ctypes.byref(h), 16, dt, 16, 0.3, 0.3, B, n, V, 16, 16, None, ws, 1 << 30, None)
    assert L.dels_draft_block(*args(200, 16, 151936)) == -2          # B > 128
    assert L.dels_draft_block(*args(4, 0, 151936)) == -2             # n < 1
    assert L.dels_draft_block(*args(4, 33, 151936)) == -2            # n > 32
    assert L.dels_draft_block(*args(4, 16, 1001)) == -2              # V % 8 != 0
    assert L.dels_draft_block(*args(4, 16, 151936, dt=5)) == -3      # logit dtype
    h.w[1] = None
    assert L.dels_draft_block(*args(4, 16, 151936)) == -1            # missing W_hh
    h.w[1] = 40
    assert L.dels_draft_block(*args(4, 16, 151936)) == -4            # misaligned W_hh
    h.w[1] = 32
    h.d_rank = 100
    assert L.dels_draft_block(*args(4, 16, 151936)) == -2            # bf16 dims must be multiples of 16
    h.d_rank = 256
    h.kind = 2
    h.wdtype = 0
    assert L.dels_draft_block(*args(4, 16, 151936)) == -6            # f32 transformer head unsupported
    assert L.dels_draft_workspace_bytes(ctypes.byref(h), 4, 16, 151936) == 0


def test_weighted_draft_rejects_bad_weights_before_enqueueing(dels):
    L = dels.lib()
    h = dels.LocalHead()
    n = 4
    good = (ctypes.c_float * n)(0.0, 0.5, 0.5, 0.5)
    bad = (ctypes.c_float * n)(0.0, float("nan"), 0.5, 0.5)
    args = lambda a, b, nn: (ctypes.byref(h), None, 0, None, a, b, 1, nn, 64, None, None, None, None, 0, None)
    assert L.dels_draft_block_weighted(*args(None, ctypes.cast(good, ctypes.c_void_p), n)) == -1
    assert L.dels_draft_block_weighted(*args(ctypes.cast(good, ctypes.c_void_p), ctypes.cast(bad, ctypes.c_void_p),
                                             n)) == -2
    assert L.dels_draft_block_weighted(*args(ctypes.cast(good, ctypes.c_void_p), ctypes.cast(good, ctypes.c_void_p),
                                             0)) == -2


def test_prior_entry_points_reject_bad_arguments_before_enqueueing(dels):
    L = dels.lib()
    V = 1000
    assert dels.dels_prior_workspace_bytes(0, 10) == 0
    assert dels.dels_prior_workspace_bytes(V, -1) == 0
    need = 1 << 16                                  # enough for every check below to come first
    ws = ctypes.create_string_buffer(need + 16)
    wsp = (ctypes.addressof(ws) + 15) // 16 * 16
    buf = ctypes.create_string_buffer(1 << 16)
    p = (ctypes.addressof(buf) + 15) // 16 * 16
    # dels_prior_count(tokens, mask, N, V, counts, tally, ws, bytes, stream)
    assert L.dels_prior_count(p, p, -1, V, p, None, wsp, need, None) == -2
    assert L.dels_prior_count(p, p, 10, 0, p, None, wsp, need, None) == -2
    assert L.dels_prior_count(None, p, 10, V, p, None, wsp, need, None) == -1
    assert L.dels_prior_count(p, None, 10, V, p, None, wsp, need, None) == -1
    assert L.dels_prior_count(p, p, 10, V, None, None, wsp, need, None) == -1
    assert L.dels_prior_count(p + 2, p, 10, V, p, None, wsp, need, None) == -4     # ids not 4-byte aligned
    assert L.dels_prior_count(p, p, 10, V, p + 4, None, wsp, need, None) == -4     # counts not 8-byte aligned
    assert L.dels_prior_count(p, p, 10, V, p, None, None, need, None) == -5
    assert L.dels_prior_count(p, p, 10, V, p, None, wsp, 100, None) == -5
    assert L.dels_prior_count(None, None, 0, V, p, None, wsp, need, None) == 0    # empty corpus: nothing to do
    # dels_prior_log(counts, V, lambda, out, ws, bytes, stream)
    for lam in (0.0, -1.0, float("inf"), float("nan")):
        assert L.dels_prior_log(p, V, lam, p, wsp, need, None) == -2
    assert L.dels_prior_log(None, V, 1.0, p, wsp, need, None) == -1
    assert L.dels_prior_log(p, V, 1.0, None, wsp, need, None) == -1
    assert L.dels_prior_log(p, V, 1.0, p, wsp, 256 + 8 * V - 1, None) == -5
    # dels_prior_estimate(tokens, mask, N, V, lambda, out, counts, tally, ws, bytes, stream)
    assert L.dels_prior_estimate(p, p, 10, V, 0.0, p, None, None, wsp, need, None) == -2
    assert L.dels_prior_estimate(p, p, 10, V, 1.0, None, None, None, wsp, need, None) == -1
    assert L.dels_prior_estimate(p, p, 10, V, 1.0, p, p + 4, None, wsp, need, None) == -4
    assert L.dels_prior_estimate(p, p, 10, V, 1.0, p, None, None, wsp, 256 + 8 * V - 1, None) == -5


def test_sampled_entry_points_reject_bad_arguments_before_enqueueing(dels):
    L = dels.lib()
    buf0 = ctypes.create_string_buffer(64)
    head = dels.LocalHead()
    head.kind, head.wdtype, head.d_model, head.d_hidden, head.d_rank = 0, 1, 64, 64, 64
    head.w_vocab = (ctypes.addressof(buf0) + 15) // 16 * 16
    buf = ctypes.create_string_buffer(1 << 16)
    p = (ctypes.addressof(buf) + 15) // 16 * 16
    w = (ctypes.c_float * 4)(0.5, 0.5, 0.5, 0.5)
    bad = (ctypes.c_float * 4)(0.5, float("nan"), 0.5, 0.5)
    hp = ctypes.byref(head)
    assert dels.dels_draft_state_bytes(head, 2, 4) == 256 + 2 * 4 * 64 * 2
    assert dels.dels_draft_state_bytes(head, 2, 0) == 0
    # dels_draft_block_sampled(head, long, dt, prior, alpha, beta, B, n, V, seed, step, tok, lp, gap, state,
    #                          state_bytes, ws, ws_bytes, stream)
    args = [hp, p, 1, p, w, w, 2, 4, 1000, 1, 2, p, p, None, p, 1 << 12, p, 1 << 15, None]
    def call(**kw):
        a = list(args)
        for k, v in kw.items():
            a[int(k[1:])] = v
        return L.dels_draft_block_sampled(*a)
    assert call(_4=None) == -1                  # alpha missing
    assert call(_5=bad) == -2                   # non-finite beta
    assert call(_7=0) == -2 and call(_7=33) == -2
    assert call(_12=None) == -1                 # the logprob output is required
    assert call(_15=100) == -5                  # draft state too small
    assert call(_14=p + 4) == -4                # draft state misaligned
    # dels_verify_block_sampled(head, tok, lp, state, long, ldt, prior, alpha, beta, target, tdt, B, n, V,
    #                           seed, step, acc, bonus, gap, ws, ws_bytes, stream)
    vargs = [hp, p, p, p, p, 1, p, w, w, p, 1, 2, 4, 1000, 1, 2, p, p, None, p, 1 << 15, None]
    def vcall(**kw):
        a = list(vargs)
        for k, v in kw.items():
            a[int(k[1:])] = v
        return L.dels_verify_block_sampled(*a)
    assert vcall(_5=9) == -3 and vcall(_10=9) == -3
    assert vcall(_12=0) == -2 and vcall(_12=40) == -2
    assert vcall(_8=bad) == -2
    assert vcall(_3=None) == -1                 # no draft state
    assert vcall(_16=None) == -1
    assert vcall(_19=None) == -5
    assert vcall(_3=p + 8) == -4
    assert vcall(_11=200) == -2                 # bf16 heads: B <= 128


def test_binding_refuses_host_and_strided_tensors(dels):
    """Device entry points take device pointers into dense row-major layouts:
    the binding raises before a host or strided tensor reaches the library."""
    rows, V = 2, 16
    x = torch.zeros(rows, V, dtype=torch.bfloat16)
    tok = torch.zeros(rows, dtype=torch.int32)
    f = torch.zeros(rows)
    with pytest.raises(ValueError, match="CUDA tensor"):
        dels.dels_combine_argmax(x, x, dels.DELS_BF16, None, 0.0, 0.0, rows, V, tok, f, None, None, 0)
    with pytest.raises(ValueError, match="CUDA tensor"):
        dels.dels_verify_block(tok.view(rows, 1), x, dels.DELS_BF16, rows, 1, V, tok, tok, None, None, 0)
    with pytest.raises(ValueError, match="contiguous"):
        dels._ptr(_FakeStrided())


class _FakeStrided(torch.Tensor):
    """A CUDA-looking, non-contiguous tensor (no GPU needed to build it)."""

    @staticmethod
    def __new__(cls):
        return torch.Tensor._make_subclass(cls, torch.zeros(4, 4).t())

    @property
    def is_cuda(self):
        return True
