"""Double-precision CPU oracle for the row-op family (test infrastructure
only: the tests, the smoke check and the benchmark's CPU-baseline leg use it;
the CUDA product never imports it)."""
