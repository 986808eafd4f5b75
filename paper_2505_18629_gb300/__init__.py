"""GB300-native verify step of Reflective Verification (arXiv 2505.18629).

The compute path is the C-ABI library ``librv.so`` (hand-written CUDA for
sm_103a, declared in ``include/rv.h``); ``paper_2505_18629_gb300.rv`` is its
thin ctypes binding.  ``synth`` draws seeded synthetic inputs.
"""
