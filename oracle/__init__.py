"""Fast3Dcache CPU oracle -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py`` (its CPU-baseline
leg and its ``--impl reference`` arm) may import this package.  The product
path (``paper_2511_22533_gb300``) never imports it and shares no code with
it.  ``f3dc_oracle.c`` is a plain C restatement of the paper's definitions;
this module builds it with gcc and exposes it through ctypes.
"""
from .oracle import *  # noqa: F401,F403
