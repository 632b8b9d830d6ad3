"""StepKV compression pass on GB300 (sm_103a): score -> step-reduce/fuse -> select -> compact.

The compute lives in ``libstepkv.so`` (hand-written CUDA, C ABI declared in include/stepkv.h).
This package is a thin binding: argument marshalling only.  Importing it does not load the
library; the first call does, and raises if the library has not been built.
"""
from .binding import (  # noqa: F401
    StepKVError, Params, default_params, load_library, stepkv_score, stepkv_select, stepkv_compact,
    stepkv_compress, stepkv_workspace_size, status_string, stepkv_select_static_scratch, stepkv_decode,
)
