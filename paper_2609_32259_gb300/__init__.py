"""GB300 (sm_103a) implementation of HeteroFold's prefill-free K/V transfer.

Modules:
  binding   ctypes binding of include/heterofold.h (libheterofold.so)
  pipeline  TransferJob: torch-allocated buffers + the ABI calls of a transfer
  workloads seeded synthetic inputs shaped like the paper's model pairs
  build     nvcc build of libheterofold.so (in-tree)

Importing the package loads nothing; the CUDA library is loaded on first use
and its absence is an error, never a fallback.
"""

__all__ = ["binding", "pipeline", "workloads", "build"]
