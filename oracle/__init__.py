"""CPU oracle for MM-ShiftKV prefill-only KV selection (test infrastructure).

Plain, slow, float64 numpy restatement of the method, written from the paper
(§3.2, Appendix A.4, Appendix B, Algorithm 1). It exists only to check the CUDA
path: the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg are its only users. The product library never imports, links or runs it,
and it shares no code with the CUDA path.
"""
from .mmshift_oracle import *  # noqa: F401,F403
