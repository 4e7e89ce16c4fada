"""fp64 CPU oracle for the PIFA layer -- test infrastructure only (tests/, smoke(), the bench's
CPU baseline). The product path never imports it."""
from .pifa_oracle import *  # noqa: F401,F403
from .pifa_oracle import RankDeficientError, PifaLayer, PivotInfo  # noqa: F401
