"""GB300 (sm_103a) implementation of the NormPre optimizer step.

The product is ``libnormpre.so`` (C ABI declared in ``include/normpre.h``);
``normpre`` is its ctypes binding and ``optim`` a tensor-level convenience
wrapper that only marshals torch tensors into those calls.
"""
from . import normpre  # noqa: F401
