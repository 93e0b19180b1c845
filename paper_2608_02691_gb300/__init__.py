"""GB300-native rotated INT2 paged KV cache (OptR, arXiv 2608.02691).

The compute path is the CUDA library ``liboptr.so`` built from ``csrc/``;
this package holds its thin ctypes binding (``optr``), the build step
(``build``) and the seeded synthetic inputs (``synth``).  Importing the
package loads nothing; the first call through ``optr`` loads the library and
raises if it has not been built.
"""
