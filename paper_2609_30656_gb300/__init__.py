"""GB300-native pooled embedding-bag (table-batched embedding) forward and backward.

The compute runs in hand-written CUDA kernels for sm_103a behind the C ABI in
``include/cb_tbe.h`` (library ``libcb_tbe.so`` in this package). ``tbe.TBE`` is
the thin Python binding over that ABI; ``workloads`` draws seeded synthetic
inputs. Importing this package does not load the CUDA library; constructing a
``TBE`` does, and fails loudly if the library has not been built.
"""

__all__ = ["workloads", "tbe"]
