"""fp64 CPU oracle for thin-key attention: TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU legs of
``bench.py`` (``cpu_baseline`` and ``--impl reference``) may import this
package.  It shares no code with the CUDA library and never imports it.

Modules:
  attention  -- per-head softmax attention (paper Section 2.1, Eqs. 1-4):
                prefill (causal or not), single-token decode, paged gather.
  cache      -- reference cache append (contiguous / paged) and the int8
                per-token absmax key quantiser.
  brute      -- pure-Python brute force used to pin ``attention``.
"""
from . import attention, brute, cache  # noqa: F401
