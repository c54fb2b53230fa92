"""fp64 CPU oracle of the STaR-KV compression stage.

TEST INFRASTRUCTURE: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import it.
The CUDA library never imports, links or runs anything from here.
"""
from .starkv_oracle import *  # noqa: F401,F403
from .starkv_oracle import Params, LayerState  # noqa: F401
