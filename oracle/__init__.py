"""CPU oracle for the Monte Carlo mutation-selection (MCA) trial loop.

TEST INFRASTRUCTURE ONLY. This package is a plain, slow, fp64 restatement of the method, used to
check the CUDA path. Only the tests, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import it. The product path (the C-ABI library and
its Python binding) never imports, links or calls anything in here, and it shares no code with it.
"""
from .mca_oracle import *  # noqa: F401,F403
from .mca_tfm import *  # noqa: F401,F403
