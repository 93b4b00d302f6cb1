"""GB300-native batched candidate-plan pricing (Heddle's planner hot path).

The CUDA library ``libheddle.so`` (C ABI, ``include/heddle.h``) does all the
work; ``heddle`` is its thin ctypes binding and ``workloads`` builds seeded
synthetic inputs.  Importing the package loads nothing; the binding loads the
library on first use and raises if it is missing.
"""
