"""GB300-native keyed Poisson-race multi-draft speculative sampler.

The compute path is the C-ABI library ``libpps.so`` (hand-written CUDA for
sm_103a, sources in ``csrc/``); :mod:`paper_2609_21858_gb300.pps` is a thin
ctypes binding with the same entry-point names.  :mod:`.synth` draws the
seeded synthetic workloads.  Importing the package loads nothing native; the
first call into :mod:`.pps` loads the library and raises if it is missing.
"""
__all__ = ["pps", "synth"]
