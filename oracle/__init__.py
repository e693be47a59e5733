"""CPU oracle of the RippleKV serving path: test infrastructure only.

Only tests, the smoke check and the benchmark's CPU-baseline leg import it.
"""
