"""GB300 (sm_103a) implementation of GRKV's prefill-time KV-cache compression.

The compute path is the CUDA library libgrkv.so (C ABI in include/grkv.h);
`binding` is its thin ctypes binding and `api` the torch-facing helpers.
"""
