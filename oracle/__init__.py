"""CPU oracle of the HeadKV decode path (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may
import this package. The product path (paper_2605_20600_gb300) never does.
"""
from . import headkv  # noqa: F401
