"""GB300 (sm_103a) policy-loss library for black-box agent RL (arXiv 2608.16798).

The compute path is the C-ABI library ``librl_loss.so`` (CUDA kernels under
``csrc/``, declared in ``include/rl_loss.h``); ``rl_loss`` is its thin Python
binding and ``build`` compiles it. Importing this package loads nothing; the
binding loads the library on first use and raises if it has not been built.
"""

__all__ = ["build", "rl_loss", "workloads"]
