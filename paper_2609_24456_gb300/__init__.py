"""libedp: a GB300-native hot path for an Experience Data Plane.

Submodules:
  edp       -- thin ctypes binding of the C ABI (include/edp.h)
  build     -- nvcc build of libedp.so for sm_103a
  fixtures  -- seeded synthetic inputs (no method arithmetic)

Importing the package loads nothing; ``edp.lib()`` loads libedp.so on first
use and raises when it has not been built.
"""
__all__ = ["edp", "build", "fixtures"]
