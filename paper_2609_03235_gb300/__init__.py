"""SGD-KV compression step on GB300: C-ABI library (libsgdkv) plus a thin ctypes binding.

Submodules: ``sgdkv`` (binding; loads the CUDA library on first use), ``configs``
(workload table), ``synth`` (seeded synthetic inputs).
"""
