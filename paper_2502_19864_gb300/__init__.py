"""GB300-native (sm_103a) adapter fine-tuning step of RingAda (arXiv 2502.19864).

``libringada.so`` (built from ``csrc/`` by ``build.py``) holds every kernel and the host
orchestrator behind the C ABI declared in ``include/ringada.h``; ``ringada`` is its ctypes
binding.  There is no other compute path: without the library every call raises.
"""
from . import ringada  # noqa: F401
