"""GB300-native candidate scoring for BOute's multi-objective Bayesian optimisation.

The CUDA library ``libboute.so`` (sources in ``csrc/``, C-ABI in
``include/boute.h``) holds every step of the scoring path; ``boute`` is its thin
ctypes binding. ``workloads`` draws the seeded synthetic inputs.
"""
