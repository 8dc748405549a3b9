"""CPU fp64 oracle of the eviction + decode-attention path (test infrastructure
only: imported by tests, the smoke check and the benchmark's CPU baseline,
never by the product path)."""
from .timebill_oracle import *  # noqa: F401,F403
