"""GB300 (sm_103a) verify-and-draft hot path of ReSpec (arXiv 2511.01282).

``respec``   -- ctypes binding of the C ABI in ``include/respec.h``
``pipeline`` -- ``VerifyStep``: device buffers + the four calls of one step
``build``    -- in-tree nvcc build of ``librespec.so``
"""
from . import respec  # noqa: F401
from .respec import RespecError, params  # noqa: F401
