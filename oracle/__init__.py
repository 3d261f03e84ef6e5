"""CPU oracle of the 1-bit FQT layer step (test infrastructure only).

Only `tests/`, `__graft_entry__.smoke()` and the CPU-baseline / reference leg
of `bench.py` may import this package.  It shares no code with the CUDA
library.  See `oracle/method.py` for the steps and the readings taken where
the paper is silent, and `oracle/philox.py` for the random number generator.
"""
from . import method, philox  # noqa: F401
