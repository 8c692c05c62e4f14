"""GB300-native grouped multi-tenant backbone forward with tenant-private
action heads (the group-batching hot path of JoyNexus, arXiv 2607.16074).

``jnx``      ctypes binding of the C ABI (include/jnx.h, include/jnx_ops.h)
``runtime``  PyTorch device-memory plumbing around it
``build``    builds libjnx.so for sm_103a in-tree
"""
from .jnx import JnxError, lib  # noqa: F401
