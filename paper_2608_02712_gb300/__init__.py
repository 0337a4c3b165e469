"""GB300-native numerical validation with failure forensics.

The package is a thin binding over libnmv.so (C ABI in include/nmv.h):
``validate`` / ``validate_batch`` check candidate operator outputs against
reference outputs on the GPU and return the forensic evidence (the
validation step of the paper's repair engine, Section 3.2, Eq. 1, and
Sections 4.2-4.3); ``stats`` / ``stats_batch`` record the diagnostic tensor
statistics of buffers (Section 4.2, diagnostic instrumentation).
``workloads`` holds the seeded synthetic inputs.
"""
from .nmv import (FLAGS, NmvError, Prepared, load, stats, stats_batch,  # noqa: F401
                  validate, validate_batch, validate_noalloc)
