"""GB300-native DoPR online scoring pass.

The scoring path is the C-ABI library ``libdopr.so`` (hand-written CUDA for
sm_103a, declared in ``include/dopr.h``); ``paper_2609_03311_gb300.dopr`` is
its thin ctypes binding.  ``synth`` draws the seeded synthetic inputs.
"""
__all__ = ["dopr", "synth", "build"]
