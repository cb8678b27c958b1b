"""GB300-native (sm_103a) MoARa-on-GaLore projected-Adam optimizer step.

The product is libmoara.so (C ABI in include/moara.h); ``binding`` is its
ctypes binding and ``buffers`` holds torch-allocated device buffers for it.
Importing the package fails if the library has not been built.
"""

from . import binding
from .binding import *  # noqa: F401,F403  (the C entry points, same names)
from .buffers import ModuleBuffers, MoaraGroup

__all__ = ["binding", "ModuleBuffers", "MoaraGroup"] + binding.EXPORTED
