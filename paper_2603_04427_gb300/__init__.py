"""Thin-key ("factored-key") attention for GB300 (sm_103a).

The compute runs in the CUDA library ``libtk.so`` behind the C ABI declared
in ``include/tk.h``; ``binding`` marshals torch tensors into those calls.
Importing this package does not load the library; the first binding call
does, and raises if it is missing.
"""
