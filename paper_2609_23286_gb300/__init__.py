"""GB300-native regulated streaming attention (RegVGGT hot path).

The compute path is the C-ABI library ``libregmem.so`` built from ``csrc/``;
``regmem`` is its thin ctypes binding.  Importing this package does not load
the library; ``regmem.load()`` does, and fails loudly when it is missing.
"""
__all__ = ["regmem", "synth"]
