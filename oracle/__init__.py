"""Plain CPU oracle of the region-sparse DiT step (RegionCache).

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports this package:
only the test suite, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` call it.  It shares no code with the
CUDA library; both sides read the same seeded inputs from
``paper_2608_29809_gb300.synth``.
"""
from .regioncache import *  # noqa: F401,F403
