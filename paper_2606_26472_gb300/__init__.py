"""EpiKV eviction hot path for GB300 (sm_103a): a C-ABI CUDA library
(libepikv.so, include/epikv.h) and its thin Python binding."""
from . import epikv  # noqa: F401
