"""GB300-native Whisper-Flash speculative decode step.

The compute path lives in the CUDA library built from `csrc/` (a C-ABI shared
object, `libwf.so`); `binding` marshals arguments to it.  `synthetic` draws the
seeded inputs.  Importing this package loads nothing: the binding loads the
library on first use and raises if it is missing.
"""
__all__ = ["binding", "synthetic"]
