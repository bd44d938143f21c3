"""GB300-native hot path of the Aladdin scheduler (arxiv 2405.06856).

Batched SLO-feasibility scoring of candidate (query, worker) placements, greedy
best-fit placement rounds (Algorithm 1) and the minimum-worker search, as CUDA
kernels for sm_103a behind a C ABI (``include/aladdin.h``).

Importing the package loads nothing; ``paper_2405_06856_gb300.aladdin`` loads
the compiled library and raises if it is missing. ``synth`` holds the seeded
workload generators and no scheduling arithmetic.
"""
