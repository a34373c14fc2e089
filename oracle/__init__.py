"""fp64 CPU oracle for the policy-update path (test infrastructure only).

Only the tests, the package entry file's smoke check and the benchmark's CPU
baseline leg may import this package; the CUDA library never does.
"""
from .molt_oracle import *  # noqa: F401,F403
