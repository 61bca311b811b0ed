"""GB300-native (sm_103a) rollout / re-scoring hot path of VLA-RL (arXiv 2505.18719).

The product is the C-ABI library ``libvla.so`` (CUDA, built from ``csrc/``) declared in
``include/vla.h``; ``paper_2505_18719_gb300.vla`` is its thin ctypes binding.
"""
