"""fp64 CPU oracle of the verifier hot path -- TEST INFRASTRUCTURE ONLY.

Imported by the tests, the smoke check and the benchmark's CPU-baseline leg;
never by the product package.
"""
