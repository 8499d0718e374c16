"""GB300-native OffQ W4A4 linear path: C-ABI library (liboffq.so) + Python binding."""

from .offq import *  # noqa: F401,F403
from .offq import OffqError, load_library, library_path, declared_symbols  # noqa: F401
