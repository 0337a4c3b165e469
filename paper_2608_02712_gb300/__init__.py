"""GB300-native numerical validation with failure forensics.

The package is a thin binding over libnmv.so (C ABI in include/nmv.h):
``validate`` / ``validate_batch`` check candidate operator outputs against
reference outputs on the GPU and return the forensic evidence (the
validation step of the paper's repair engine, Section 3.2, Eq. 1, and
Sections 4.2-4.3); ``stats`` / ``stats_batch`` record the diagnostic tensor
statistics of buffers (Section 4.2, diagnostic instrumentation);
``forensics`` / ``forensics_batch`` the ulp distances, fp16-ceiling counts,
error growth and per-axis maps behind the scheduling rules (Section 4.4);
``sweep`` the full-coverage escalation with its sealed evidence record
(Section 4.3).
``workloads`` holds the seeded synthetic inputs.
"""
from .nmv import (FLAGS, FX_FLAGS, NmvError, Prepared, PreparedSweep, forensics, forensics_batch,  # noqa: F401
                  load, sha256, stats, stats_batch, sweep, validate, validate_batch,
                  validate_noalloc)
