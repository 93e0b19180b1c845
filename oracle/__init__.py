"""Test infrastructure: the fp64 CPU oracle of the rotated INT2 paged
KV-cache path.  Only the tests, the smoke check and the benchmark's CPU
baseline may import it; the CUDA library never does."""
