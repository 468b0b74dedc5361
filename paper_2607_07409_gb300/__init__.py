"""Python binding of ``libdels.so``, the DeLS-Spec drafting hot path on GB300.

Argument marshalling only: every step of the drafting loop, the combine and
the verification runs in the library's CUDA kernels. Functions named
``dels_*`` mirror the C ABI in ``include/dels.h`` one to one and take torch
tensors (or raw integer device pointers) in place of the C pointers. The
``Drafter`` helper keeps a local head's weight pointers and a workspace for
repeated calls. There is no CPU fallback: if ``libdels.so`` has not been
built, every call raises ``RuntimeError``.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional

import torch

__all__ = [
    "DELS_OK", "DELS_F32", "DELS_BF16",
    "DELS_HEAD_GRU", "DELS_HEAD_MLP", "DELS_HEAD_XFMR", "DELS_HEAD_MARKOV",
    "DELS_STATUS_NONFINITE", "DELS_STATUS_TIMEOUT", "DELS_STATUS_BAD_TOKEN",
    "DELS_ERR_NULL_POINTER", "DELS_ERR_BAD_SHAPE", "DELS_ERR_BAD_DTYPE", "DELS_ERR_ALIGNMENT",
    "DELS_ERR_WORKSPACE", "DELS_ERR_UNSUPPORTED", "DELS_ERR_CUDA", "DELS_ERR_TOO_LARGE",
    "DelsError", "LocalHead", "lib", "library_path", "exported_symbols",
    "dels_draft_workspace_bytes", "dels_draft_block", "dels_draft_block_weighted",
    "dels_draft_state_bytes", "dels_draft_block_sampled",
    "dels_verify_sampled_workspace_bytes", "dels_verify_block_sampled",
    "dels_combine_workspace_bytes", "dels_combine_argmax", "dels_combine_argmax_noalloc",
    "dels_verify_workspace_bytes", "dels_verify_block",
    "dels_read_status", "dels_prior_from_counts", "dels_status_string", "dels_version",
    "dels_profile_enable", "dels_profile_reset", "dels_profile_read", "KCLASS",
    "dels_gru_input_table_bytes", "dels_gru_build_input_table", "gru_input_table",
    "dels_selftest_timeout_bytes", "dels_selftest_timeout", "dels_selftest_gumbel",
    "dels_prior_workspace_bytes", "dels_prior_count", "dels_prior_log", "dels_prior_estimate", "estimate_prior",
    "make_head", "Drafter", "dtype_code",
]

DELS_OK = 0
DELS_F32, DELS_BF16 = 0, 1
DELS_HEAD_GRU, DELS_HEAD_MLP, DELS_HEAD_XFMR, DELS_HEAD_MARKOV = 0, 1, 2, 3
DELS_STATUS_NONFINITE, DELS_STATUS_TIMEOUT, DELS_STATUS_BAD_TOKEN = 1, 2, 4
(DELS_ERR_NULL_POINTER, DELS_ERR_BAD_SHAPE, DELS_ERR_BAD_DTYPE, DELS_ERR_ALIGNMENT, DELS_ERR_WORKSPACE,
 DELS_ERR_UNSUPPORTED, DELS_ERR_CUDA, DELS_ERR_TOO_LARGE) = -1, -2, -3, -4, -5, -6, -7, -8

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libdels.so")
_lib = None

# name -> (restype, argtypes); the C ABI of include/dels.h
_vp, _i, _f, _d, _sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_double, ctypes.c_size_t


class LocalHead(ctypes.Structure):
    """Mirror of ``dels_local_head``."""

    _fields_ = [
        ("kind", ctypes.c_int), ("wdtype", ctypes.c_int),
        ("d_model", ctypes.c_int), ("d_hidden", ctypes.c_int), ("d_rank", ctypes.c_int),
        ("window", ctypes.c_int), ("n_layers", ctypes.c_int), ("n_heads", ctypes.c_int),
        ("max_pos", ctypes.c_int),
        ("emb", ctypes.c_void_p), ("w", ctypes.c_void_p * 8), ("w_vocab", ctypes.c_void_p),
    ]


_SIGS = {
    "dels_selftest_timeout_bytes": (_sz, []),
    "dels_selftest_timeout": (_i, [_vp, _sz, _vp]),
    "dels_selftest_gumbel": (_i, [_vp, _vp, ctypes.c_longlong, _vp]),
    "dels_gru_input_table_bytes": (_sz, [ctypes.POINTER(LocalHead), _i]),
    "dels_gru_build_input_table": (_i, [ctypes.POINTER(LocalHead), _i, _vp, _sz, _vp, _sz, _vp]),
    "dels_draft_workspace_bytes": (_sz, [ctypes.POINTER(LocalHead), _i, _i, _i]),
    "dels_draft_block": (_i, [ctypes.POINTER(LocalHead), _vp, _i, _vp, _f, _f, _i, _i, _i, _vp, _vp, _vp, _vp, _sz,
                              _vp]),
    "dels_draft_block_weighted": (_i, [ctypes.POINTER(LocalHead), _vp, _i, _vp, _vp, _vp, _i, _i, _i, _vp, _vp, _vp,
                                       _vp, _sz, _vp]),
    "dels_draft_state_bytes": (_sz, [ctypes.POINTER(LocalHead), _i, _i]),
    "dels_draft_block_sampled": (_i, [ctypes.POINTER(LocalHead), _vp, _i, _vp, _vp, _vp, _i, _i, _i, ctypes.c_uint64,
                                      ctypes.c_uint64, _vp, _vp, _vp, _vp, _sz, _vp, _sz, _vp]),
    "dels_verify_sampled_workspace_bytes": (_sz, [ctypes.POINTER(LocalHead), _i, _i, _i, _i]),
    "dels_verify_block_sampled": (_i, [ctypes.POINTER(LocalHead), _vp, _vp, _vp, _vp, _i, _vp, _vp, _vp, _vp, _i, _i,
                                       _i, _i, ctypes.c_uint64, ctypes.c_uint64, _vp, _vp, _vp, _vp, _sz, _vp]),
    "dels_combine_workspace_bytes": (_sz, [_i, _i, _i]),
    "dels_combine_argmax": (_i, [_vp, _vp, _i, _vp, _f, _f, _i, _i, _vp, _vp, _vp, _vp, _sz, _vp]),
    "dels_combine_argmax_noalloc": (_i, [_vp, _vp, _i, _vp, _f, _f, _i, _i, _vp, _vp, _vp, _vp]),
    "dels_verify_workspace_bytes": (_sz, [_i, _i, _i, _i]),
    "dels_verify_block": (_i, [_vp, _vp, _i, _i, _i, _i, _vp, _vp, _vp, _vp, _sz, _vp]),
    "dels_read_status": (_i, [_vp, _vp, ctypes.POINTER(ctypes.c_int32)]),
    "dels_prior_from_counts": (_i, [_vp, _i, _d, _vp]),
    "dels_prior_workspace_bytes": (_sz, [_i, ctypes.c_int64]),
    "dels_prior_count": (_i, [_vp, _vp, ctypes.c_int64, _i, _vp, _vp, _vp, _sz, _vp]),
    "dels_prior_log": (_i, [_vp, _i, _d, _vp, _vp, _sz, _vp]),
    "dels_prior_estimate": (_i, [_vp, _vp, ctypes.c_int64, _i, _d, _vp, _vp, _vp, _vp, _sz, _vp]),
    "dels_status_string": (ctypes.c_char_p, [_i]),
    "dels_version": (_i, []),
    "dels_profile_enable": (_i, [_i]),
    "dels_profile_reset": (_i, []),
    "dels_profile_read": (_i, [_i, ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_double)]),
}

# kernel classes of the optional profiler
KCLASS = {"vocab_combine": 0, "head_gemm": 1, "head_misc": 2, "merge": 3, "pos0": 4, "verify": 5, "combine": 6,
          "draft_block": 7, "prior": 8}


def exported_symbols():
    """Names of the C ABI entry points this binding expects the library to export."""
    return list(_SIGS)


class DelsError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {dels_status_string(code)} ({code})")


def library_path() -> str:
    return _LIB_PATH


def lib():
    """The loaded ``libdels.so`` (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(
                f"{_LIB_PATH} not found: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(_LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


# ----------------------------------------------------------------------------- marshalling helpers

def _ptr(x) -> Optional[int]:
    """Device address of a CUDA tensor, or an integer address passed through.

    Every pointer the library's entry points take through this helper is a
    device pointer into a row-major layout, so a host tensor or a strided
    view is refused here instead of reaching a kernel."""
    if x is None:
        return None
    if isinstance(x, torch.Tensor):
        if not x.is_cuda:
            raise ValueError("expected a CUDA tensor: the library's entry points take device pointers")
        if not x.is_contiguous():
            raise ValueError("expected a contiguous tensor: the library's layouts are dense row-major")
        return x.data_ptr()
    return int(x)


def _stream(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream if torch.cuda.is_available() else None
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def dtype_code(t) -> int:
    if isinstance(t, torch.Tensor):
        t = t.dtype
    if t == torch.float32:
        return DELS_F32
    if t == torch.bfloat16:
        return DELS_BF16
    raise ValueError(f"unsupported dtype {t}")


def _check(code: int, where: str):
    if code != DELS_OK:
        raise DelsError(code, where)


# ----------------------------------------------------------------------------- the C ABI, by name

def dels_version() -> int:
    return lib().dels_version()


def dels_status_string(code: int) -> str:
    return lib().dels_status_string(int(code)).decode()


def dels_selftest_timeout_bytes() -> int:
    return lib().dels_selftest_timeout_bytes()


def dels_selftest_timeout(workspace, workspace_bytes: int, stream=None) -> int:
    return lib().dels_selftest_timeout(_ptr(workspace), workspace_bytes, _stream(stream))


def dels_selftest_gumbel(bits, g, n: int, stream=None) -> int:
    return lib().dels_selftest_gumbel(_ptr(bits), _ptr(g), n, _stream(stream))


def dels_gru_input_table_bytes(head: LocalHead, V: int) -> int:
    return lib().dels_gru_input_table_bytes(ctypes.byref(head), V)


def dels_gru_build_input_table(head: LocalHead, V: int, table, table_bytes: int, workspace, workspace_bytes: int,
                               stream=None) -> int:
    return lib().dels_gru_build_input_table(ctypes.byref(head), V, _ptr(table), table_bytes, _ptr(workspace),
                                            workspace_bytes, _stream(stream))


def gru_input_table(spec, weights: Dict[str, torch.Tensor], V: int, stream=None) -> torch.Tensor:
    """The GRU input table G = E W_ih^T [V, 3*d_hidden] float32 of a bf16 GRU
    head, built on the weights' device. Put it in the weights dict as
    ``input_table`` to have dels_draft_block read it."""
    head = make_head(spec, {k: v for k, v in weights.items() if k != "input_table"})
    nbytes = dels_gru_input_table_bytes(head, V)
    if nbytes == 0:
        raise DelsError(-6, "dels_gru_input_table_bytes")
    dev = weights["emb"].device
    table = torch.empty(nbytes // 4, dtype=torch.float32, device=dev).view(V, -1)
    ws = torch.zeros(256, dtype=torch.uint8, device=dev)
    _check(dels_gru_build_input_table(head, V, table, nbytes, ws, 256, stream), "dels_gru_build_input_table")
    st = dels_read_status(ws, stream)
    if st != 0:
        raise DelsError(st, "dels_gru_build_input_table (device status)")
    return table


def dels_draft_workspace_bytes(head: LocalHead, B: int, n: int, V: int) -> int:
    return lib().dels_draft_workspace_bytes(ctypes.byref(head), B, n, V)


def dels_draft_block(head: LocalHead, long_logits, logit_dtype: int, log_prior, alpha: float, beta: float,
                     B: int, n: int, V: int, out_tokens, out_logprob, out_top2_gap, workspace,
                     workspace_bytes: int, stream=None) -> int:
    r = lib().dels_draft_block(ctypes.byref(head), _ptr(long_logits), logit_dtype, _ptr(log_prior), alpha, beta,
                               B, n, V, _ptr(out_tokens), _ptr(out_logprob), _ptr(out_top2_gap),
                               _ptr(workspace), workspace_bytes, _stream(stream))
    return r


def dels_draft_block_weighted(head: LocalHead, long_logits, logit_dtype: int, log_prior, alpha, beta, B: int,
                              n: int, V: int, out_tokens, out_logprob, out_top2_gap, workspace,
                              workspace_bytes: int, stream=None) -> int:
    """Per-position fusion weights: ``alpha``/``beta`` are sequences of n floats
    (host; entry 0 unused)."""
    a = (ctypes.c_float * n)(*[float(x) for x in alpha])
    b = (ctypes.c_float * n)(*[float(x) for x in beta])
    return lib().dels_draft_block_weighted(ctypes.byref(head), _ptr(long_logits), logit_dtype, _ptr(log_prior),
                                           ctypes.cast(a, ctypes.c_void_p), ctypes.cast(b, ctypes.c_void_p), B, n, V,
                                           _ptr(out_tokens), _ptr(out_logprob), _ptr(out_top2_gap),
                                           _ptr(workspace), workspace_bytes, _stream(stream))


def _host_floats(xs, n):
    xs = [float(x) for x in xs]
    if len(xs) != n:
        raise ValueError(f"expected {n} per-position weights")
    arr = (ctypes.c_float * n)(*xs)
    return arr, ctypes.cast(arr, ctypes.c_void_p)


def dels_draft_state_bytes(head: LocalHead, B: int, n: int) -> int:
    return lib().dels_draft_state_bytes(ctypes.byref(head), B, n)


def dels_draft_block_sampled(head: LocalHead, long_logits, logit_dtype: int, log_prior, alpha, beta, B: int, n: int,
                             V: int, seed: int, step: int, out_tokens, out_logprob, out_key_gap, draft_state,
                             state_bytes: int, workspace, workspace_bytes: int, stream=None) -> int:
    """Temperature-1 drafting; ``alpha``/``beta`` are sequences of n floats (host)."""
    a, ap = _host_floats(alpha, n)
    b, bp = _host_floats(beta, n)
    return lib().dels_draft_block_sampled(ctypes.byref(head), _ptr(long_logits), logit_dtype, _ptr(log_prior), ap, bp,
                                          B, n, V, int(seed), int(step), _ptr(out_tokens), _ptr(out_logprob),
                                          _ptr(out_key_gap), _ptr(draft_state), state_bytes, _ptr(workspace),
                                          workspace_bytes, _stream(stream))


def dels_verify_sampled_workspace_bytes(head: LocalHead, B: int, n: int, V: int, target_dtype: int) -> int:
    return lib().dels_verify_sampled_workspace_bytes(ctypes.byref(head), B, n, V, target_dtype)


def dels_verify_block_sampled(head: LocalHead, draft_tokens, draft_logprob, draft_state, long_logits,
                              logit_dtype: int, log_prior, alpha, beta, target_logits, target_dtype: int, B: int,
                              n: int, V: int, seed: int, step: int, out_accept_len, out_bonus, out_bonus_gap,
                              workspace, workspace_bytes: int, stream=None) -> int:
    """Speculative-sampling verification of a temperature-1 block; ``alpha``/``beta`` host sequences of n."""
    a, ap = _host_floats(alpha, n)
    b, bp = _host_floats(beta, n)
    return lib().dels_verify_block_sampled(ctypes.byref(head), _ptr(draft_tokens), _ptr(draft_logprob),
                                           _ptr(draft_state), _ptr(long_logits), logit_dtype, _ptr(log_prior), ap, bp,
                                           _ptr(target_logits), target_dtype, B, n, V, int(seed), int(step),
                                           _ptr(out_accept_len), _ptr(out_bonus), _ptr(out_bonus_gap),
                                           _ptr(workspace), workspace_bytes, _stream(stream))


def dels_combine_workspace_bytes(rows: int, V: int, dtype: int) -> int:
    return lib().dels_combine_workspace_bytes(rows, V, dtype)


def dels_combine_argmax(long_logits, short_logits, dtype: int, log_prior, alpha: float, beta: float, rows: int,
                        V: int, out_token, out_logprob, out_top2_gap, workspace, workspace_bytes: int,
                        stream=None) -> int:
    return lib().dels_combine_argmax(_ptr(long_logits), _ptr(short_logits), dtype, _ptr(log_prior), alpha, beta,
                                     rows, V, _ptr(out_token), _ptr(out_logprob), _ptr(out_top2_gap),
                                     _ptr(workspace), workspace_bytes, _stream(stream))


def dels_combine_argmax_noalloc(long_logits, short_logits, dtype: int, log_prior, alpha: float, beta: float,
                                rows: int, V: int, out_token, out_logprob, out_top2_gap, stream=None) -> int:
    """dels_combine_argmax without a workspace: uses the library's fixed 4 MiB
    device scratch (for callers that cannot allocate device memory)."""
    return lib().dels_combine_argmax_noalloc(_ptr(long_logits), _ptr(short_logits), dtype, _ptr(log_prior), alpha,
                                             beta, rows, V, _ptr(out_token), _ptr(out_logprob), _ptr(out_top2_gap),
                                             _stream(stream))


def dels_verify_workspace_bytes(B: int, n: int, V: int, dtype: int) -> int:
    return lib().dels_verify_workspace_bytes(B, n, V, dtype)


def dels_verify_block(draft_tokens, target_logits, dtype: int, B: int, n: int, V: int, out_accept_len, out_bonus,
                      out_target_argmax, workspace, workspace_bytes: int, stream=None) -> int:
    return lib().dels_verify_block(_ptr(draft_tokens), _ptr(target_logits), dtype, B, n, V, _ptr(out_accept_len),
                                   _ptr(out_bonus), _ptr(out_target_argmax), _ptr(workspace), workspace_bytes,
                                   _stream(stream))


def dels_read_status(workspace, stream=None) -> int:
    out = ctypes.c_int32(0)
    _check(lib().dels_read_status(_ptr(workspace), _stream(stream), ctypes.byref(out)), "dels_read_status")
    return out.value


def dels_prior_from_counts(counts: torch.Tensor, lam: float = 1.0) -> torch.Tensor:
    """Host helper: float32 log prior [V] from int64 counts [V] (both CPU tensors)."""
    c = counts.detach().to("cpu", torch.int64).contiguous()
    out = torch.empty(c.numel(), dtype=torch.float32)
    _check(lib().dels_prior_from_counts(c.data_ptr(), c.numel(), float(lam), out.data_ptr()),
           "dels_prior_from_counts")
    return out


def dels_prior_workspace_bytes(V: int, N: int) -> int:
    return lib().dels_prior_workspace_bytes(V, N)


def dels_prior_count(tokens, loss_mask, N: int, V: int, counts, tally, workspace, workspace_bytes: int,
                     stream=None) -> int:
    """counts/tally: int64 (uint64 bit pattern) device tensors, accumulated."""
    return lib().dels_prior_count(_ptr(tokens), _ptr(loss_mask), N, V, _ptr(counts), _ptr(tally), _ptr(workspace),
                                  workspace_bytes, _stream(stream))


def dels_prior_log(counts, V: int, lam: float, out_log_prior, workspace, workspace_bytes: int, stream=None) -> int:
    return lib().dels_prior_log(_ptr(counts), V, float(lam), _ptr(out_log_prior), _ptr(workspace), workspace_bytes,
                                _stream(stream))


def dels_prior_estimate(tokens, loss_mask, N: int, V: int, lam: float, out_log_prior, out_counts, out_tally,
                        workspace, workspace_bytes: int, stream=None) -> int:
    return lib().dels_prior_estimate(_ptr(tokens), _ptr(loss_mask), N, V, float(lam), _ptr(out_log_prior),
                                     _ptr(out_counts), _ptr(out_tally), _ptr(workspace), workspace_bytes,
                                     _stream(stream))


def estimate_prior(tokens: torch.Tensor, loss_mask: torch.Tensor, V: int, lam: float = 1.0, stream=None):
    """Device unigram prior of a corpus: (log prior float32 [V], counts int64 [V],
    tally int64 [2] = positions counted, loss-masked ids outside [0, V))."""
    if tokens.dtype != torch.int32 or loss_mask.dtype not in (torch.uint8, torch.bool):
        raise ValueError("tokens must be int32 and loss_mask uint8")
    if tokens.numel() != loss_mask.numel():
        raise ValueError("tokens and loss_mask must have the same length")
    if not (tokens.is_contiguous() and loss_mask.is_contiguous()):
        raise ValueError("tokens and loss_mask must be contiguous")
    dev = tokens.device
    nbytes = dels_prior_workspace_bytes(V, tokens.numel())
    if nbytes == 0:
        raise DelsError(-2, "dels_prior_workspace_bytes")
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=dev)
    out = torch.empty(V, dtype=torch.float32, device=dev)
    counts = torch.empty(V, dtype=torch.int64, device=dev)
    tally = torch.empty(2, dtype=torch.int64, device=dev)
    _check(dels_prior_estimate(tokens, loss_mask.view(torch.uint8), tokens.numel(), V, lam, out, counts, tally, ws,
                               nbytes, stream), "dels_prior_estimate")
    return out, counts, tally


def dels_profile_enable(on: bool) -> None:
    _check(lib().dels_profile_enable(1 if on else 0), "dels_profile_enable")


def dels_profile_reset() -> None:
    _check(lib().dels_profile_reset(), "dels_profile_reset")


def dels_profile_read(kernel_class: int):
    """(launches, total device ms) of one kernel class since the last reset."""
    n = ctypes.c_int(0)
    ms = ctypes.c_double(0.0)
    _check(lib().dels_profile_read(int(kernel_class), ctypes.byref(n), ctypes.byref(ms)), "dels_profile_read")
    return n.value, ms.value


# ----------------------------------------------------------------------------- conveniences

_KIND = {"gru": DELS_HEAD_GRU, "mlp": DELS_HEAD_MLP, "xfmr": DELS_HEAD_XFMR, "markov": DELS_HEAD_MARKOV}
_SLOTS = {
    "gru": ["w_ih", "w_hh", "w_rank", "input_table"],
    "mlp": ["w1", "w2"],
    "xfmr": ["pos", "wq", "wk", "wv", "wo", "w1", "w2"],
    "markov": [],
}


def make_head(spec, weights: Dict[str, torch.Tensor]) -> LocalHead:
    """LocalHead for a head spec (``kind``, ``wdtype``, dims) and a dict of device weight tensors
    (keys emb, w_vocab and the kind's slot names). The caller keeps the tensors alive."""
    h = LocalHead()
    h.kind = _KIND[spec.kind]
    h.wdtype = DELS_BF16 if spec.wdtype == "bf16" else DELS_F32
    h.d_model, h.d_hidden, h.d_rank = spec.d_model, spec.d_hidden, spec.d_rank
    h.window, h.n_layers, h.n_heads, h.max_pos = spec.window, spec.n_layers, spec.n_heads, spec.max_pos
    h.emb = _ptr(weights["emb"])
    h.w_vocab = _ptr(weights["w_vocab"])
    for i, name in enumerate(_SLOTS[spec.kind]):
        if name in weights:
            h.w[i] = _ptr(weights[name])
    return h


class Drafter:
    """One local head + one workspace for repeated dels_draft_block calls."""

    def __init__(self, spec, weights: Dict[str, torch.Tensor], B: int, n: int, V: int, device=None):
        self.spec, self.weights = spec, weights
        self.head = make_head(spec, weights)
        self.B, self.n, self.V = B, n, V
        self.device = device or weights["w_vocab"].device
        nbytes = dels_draft_workspace_bytes(self.head, B, n, V)
        if nbytes == 0:
            raise DelsError(-2, "dels_draft_workspace_bytes")
        self.ws_bytes = nbytes
        self.workspace = torch.zeros(nbytes, dtype=torch.uint8, device=self.device)
        self.tokens = torch.empty(B, n, dtype=torch.int32, device=self.device)
        self.logprob = torch.empty(B, n, dtype=torch.float32, device=self.device)
        self.gap = torch.empty(B, n, dtype=torch.float32, device=self.device)

    def __call__(self, long_logits: torch.Tensor, log_prior: torch.Tensor, alpha, beta, stream=None):
        """``alpha``/``beta``: one weight for the block, or n per-position weights."""
        if hasattr(alpha, "__len__") or hasattr(beta, "__len__"):
            a = list(alpha) if hasattr(alpha, "__len__") else [alpha] * self.n
            b = list(beta) if hasattr(beta, "__len__") else [beta] * self.n
            _check(dels_draft_block_weighted(self.head, long_logits, dtype_code(long_logits), log_prior, a, b,
                                             self.B, self.n, self.V, self.tokens, self.logprob, self.gap,
                                             self.workspace, self.ws_bytes, stream), "dels_draft_block_weighted")
        else:
            _check(dels_draft_block(self.head, long_logits, dtype_code(long_logits), log_prior, alpha, beta, self.B,
                                    self.n, self.V, self.tokens, self.logprob, self.gap, self.workspace,
                                    self.ws_bytes, stream), "dels_draft_block")
        return self.tokens, self.logprob, self.gap

    def sample(self, long_logits: torch.Tensor, log_prior: torch.Tensor, alpha, beta, seed: int, step: int,
               stream=None):
        """Temperature-1 block: returns (tokens, logprob, key gap, draft state)."""
        a = list(alpha) if hasattr(alpha, "__len__") else [alpha] * self.n
        b = list(beta) if hasattr(beta, "__len__") else [beta] * self.n
        if getattr(self, "state", None) is None:
            self.state_bytes = dels_draft_state_bytes(self.head, self.B, self.n)
            self.state = torch.zeros(self.state_bytes, dtype=torch.uint8, device=self.device)
        _check(dels_draft_block_sampled(self.head, long_logits, dtype_code(long_logits), log_prior, a, b, self.B,
                                        self.n, self.V, seed, step, self.tokens, self.logprob, self.gap, self.state,
                                        self.state_bytes, self.workspace, self.ws_bytes, stream),
               "dels_draft_block_sampled")
        return self.tokens, self.logprob, self.gap, self.state

    def status(self, stream=None) -> int:
        return dels_read_status(self.workspace, stream)
