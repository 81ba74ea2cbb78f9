"""fp64 CPU oracle for MILO decode attention and block-wise low-rank compression.

Test infrastructure only: imported by the tests, the smoke check and the
benchmark's CPU-baseline leg, never by the CUDA library."""
