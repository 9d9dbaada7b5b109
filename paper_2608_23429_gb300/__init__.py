"""GB300-native implementation of ChebBooster's online extrapolation stage.

The compute path is the C-ABI library ``libchebboost.so`` (CUDA, sm_103a),
declared in ``include/chebboost.h``; ``paper_2608_23429_gb300.chebboost`` is its
thin ctypes binding. ``workloads`` holds the seeded synthetic inputs.
"""
__version__ = "0.1.0"
