"""CPU oracle for the CacheRepair online repair path (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  The
product path (``paper_2609_35139_gb300``) never imports it and shares no code
with it.
"""
from .cacherepair import *  # noqa: F401,F403
from .offline import *  # noqa: F401,F403
from .variants import *  # noqa: F401,F403
from .training import *  # noqa: F401,F403
from .serving import *  # noqa: F401,F403
