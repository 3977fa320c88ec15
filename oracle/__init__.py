"""fp64 CPU oracle of the NormPre optimizer step.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import it.  The
CUDA library never imports, links or calls anything in this package, and this
package imports nothing from the CUDA library.
"""
from .normpre_oracle import *  # noqa: F401,F403
