"""GB300-native batch-1 decoder forward pass (prefill + paged-KV greedy decode)
behind the C ABI of include/wici.h.  `wici` is the ctypes binding; `build`
compiles libwici.so for sm_103a."""
from . import build, wici  # noqa: F401
from .wici import WiciModel, WiciError  # noqa: F401
