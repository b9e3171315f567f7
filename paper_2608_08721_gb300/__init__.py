"""LibraSpec verify round on GB300 (sm_103a).

The hot path of one LibraSpec decoding round — drafter confidence, the
marginal-gain length selector, block-causal GQA verify attention and greedy /
rejection-sampling acceptance — as hand-written CUDA kernels behind a C ABI
(``include/libraspec.h``). This package is the thin Python binding.
"""
