"""GB300-native batched AUV rollout (arXiv 2512.13359, the data-parallel
rollout step of the RL pipeline) behind a C ABI.

Importing the package does not load the CUDA library; the binding in
``paper_2512_13359_gb300.auvenv`` loads it on first use and raises if it is
missing.
"""
