"""CPU oracle of the DFlare draft path (test infrastructure only; see dflare_oracle.py)."""
from .dflare_oracle import *  # noqa: F401,F403
from .dflare_oracle import DraftOracle  # noqa: F401
