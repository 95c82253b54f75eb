"""CPU oracle for the Hadamard-domain INT8 operator. TEST INFRASTRUCTURE ONLY:
imported by tests, the smoke check and the benchmark's CPU-baseline leg, never
by the CUDA path."""
