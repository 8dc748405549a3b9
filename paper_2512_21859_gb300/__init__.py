"""GB300-native eviction + decode-attention library (TimeBill's hot path).

The compute runs in ``libtimebill_kv.so`` (hand-written CUDA for sm_103a,
C ABI declared in include/timebill_kv.h). ``binding`` wraps its entry points
with the same names; ``inputs`` draws seeded synthetic workloads. Importing
the package does not load the library: ``binding`` does, on first use, and
fails loudly if it is missing.
"""
