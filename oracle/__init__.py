"""CPU oracle of the Conduit refresh policy: test infrastructure only.

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package. It shares no code with the CUDA path.
"""

from .conduit_oracle import *  # noqa: F401,F403
