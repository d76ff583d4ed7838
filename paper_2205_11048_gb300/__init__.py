"""GBA (Global Batch gradients Aggregation, arXiv 2205.11048) aggregate-and-apply
step on GB300: a C-ABI CUDA library (``libgba.so``) and its ctypes binding.

Importing the package loads nothing; ``paper_2205_11048_gb300.binding`` loads
the library and raises if it is missing."""
