"""The fp64 CPU oracle of the Archer hot path.

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and the
CPU-baseline / reference legs of bench.py, never by the CUDA path, with which
it shares no code.
"""
