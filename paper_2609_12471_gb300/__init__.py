"""GB300-native forward pass of a Qwen3-architecture decoder (rollout decode and
teacher-forced log-prob scoring), behind the C ABI declared in include/qk.h.

Every step of the forward pass runs in the CUDA kernels of libqk.so; this
package only marshals arguments (see ``_binding``).  Importing it fails loudly
if libqk.so has not been built.
"""
from ._binding import *  # noqa: F401,F403
from ._binding import QKError, lib_path  # noqa: F401
