"""GB300-native ECOKV prefill KV-cache eviction (score -> select -> compact).

The compute path is the C-ABI library ``libecokv.so`` (hand-written sm_103a
CUDA kernels); :mod:`paper_2609_06663_gb300.ecokv` is its thin ctypes binding.
"""
