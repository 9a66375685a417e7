"""GB300-native (sm_103a) E2S-Pruner pruning decision.

The compute path lives in ``libe2s.so`` (hand-written CUDA behind a C ABI,
see ``include/e2s.h``); ``e2s`` is its ctypes binding.  Importing this
package does not load the library: ``from paper_2608_23253_gb300 import e2s``
does, and fails loudly if it has not been built.
"""
