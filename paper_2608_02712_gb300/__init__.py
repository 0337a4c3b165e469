"""GB300-native numerical validation with failure forensics.

The package is a thin binding over libnmv.so (C ABI in include/nmv.h):
``validate`` / ``validate_batch`` check candidate operator outputs against
reference outputs on the GPU and return the forensic evidence (the
validation step of the paper's repair engine, Section 3.2, Eq. 1, and
Sections 4.2-4.3).  ``workloads`` holds the seeded synthetic inputs.
"""
from .nmv import (FLAGS, NmvError, Prepared, load, validate,  # noqa: F401
                  validate_batch, validate_noalloc)
