"""CPU oracle for the DeLS-Spec per-block drafting path.

TEST INFRASTRUCTURE ONLY. This package is a plain, slow, fp64 restatement of
what the paper defines. It exists so the CUDA path can be checked against it.
Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline /
``--impl reference`` legs of ``bench.py`` may import it; the product path
(the C-ABI library and its Python binding) never does, and shares no code with
it.

What it restates (DeLS-Spec, "Decoupled Long-Short Contexts for Parallel
Speculative Drafting"):

* Section 4.3, fusion equation: l = l_L + alpha * l_S - beta * l_P.
* Algorithm 1: x_0 decoded from softmax(l_L^(0)) alone; for j = 1..s the local
  head runs over x_{0:j-1}, its logits are fused, and x_j is decoded from the
  softmax of the fused logits; the block is then verified by the target.
  Decode at temperature 0 is the argmax (lowest vocabulary index on ties);
  at temperature 1 it is a draw from the softmax by the Gumbel-max rule, with
  Philox4x32-10 uniforms, and the block is verified by lossless speculative
  sampling (accept with probability min(1, p/q), resample the residual).
* Appendix A, local heads: the RNN head (target embedding -> one bias-free GRU
  layer -> SiLU(W_rank h) -> W_vocab r) and the Markov head
  (r = E_M(x_{i-1}), l_S = W_M r).
* Appendix A, unigram prior: c(v) counts the loss-masked corpus tokens equal
  to v; p0(v) = (c(v) + lambda) / sum(c + lambda), l_P = log p0.
* Section 4.1 and Appendix B: the exact three-factor factorisation of
  p(x | y, z) (used by the tests to pin the alpha = beta = 1 case).
* Appendix D: rate_i = P(acceptance length >= i).

Readings where the paper is silent (all listed in the design notes):

* Synthetic heads for the workloads the paper does not fix: a window MLP over
  the last W drafted tokens and a 1-layer causal pre-norm transformer over the
  block prefix.
* Precision contract: weights and logits are taken exactly as stored; the
  activation vectors that feed a bf16 matrix product (the GRU state fed to
  W_hh and W_rank, the low-rank state r, MLP/transformer activations) are
  rounded to bf16 (round-to-nearest-even, through fp32) because the device
  feeds bf16 tensor-core products; everything else is fp64.

Module layout: ``core`` (prior, fusion, decode, verify, statistics,
factorisation) and ``heads`` (local heads and the block drafting loop).
"""
from .core import (  # noqa: F401
    to_f64,
    round_bf16,
    count_masked_tokens,
    log_prior,
    lse,
    fuse,
    greedy_decode,
    combine_argmax,
    verify_greedy,
    philox4x32_10,
    uniforms,
    gumbel,
    sample_decode,
    verify_sampled,
    STREAM_DRAFT,
    STREAM_ACCEPT,
    STREAM_RESIDUAL,
    acceptance_rates,
    poe_factors,
)
from .heads import (  # noqa: F401
    GruHead,
    MlpHead,
    XfmrHead,
    MarkovHead,
    make_head,
    draft_block,
    DraftResult,
)
