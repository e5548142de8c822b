"""fp64 CPU oracle of the WISE attention hot path (test infrastructure only).

Used by tests/, the smoke check and the benchmark's CPU-baseline leg; never by
the library under paper_2609_27373_gb300/, with which it shares no code.
"""
