"""GB300-native prefix-reuse prefill: paged KV restore/append and causal GQA
attention over [cached prefix ++ new tokens] (arXiv 2505.23970, Sec. 2.2).

The compute path is the CUDA library ``libgc.so`` built from ``csrc/`` for
sm_103a; ``binding`` exposes its C entry points under the same names.
"""
__all__ = ["binding", "workloads"]
