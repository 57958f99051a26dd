"""fp64 CPU oracle (test infrastructure only; never used by the library)."""
from .kvm_oracle import *  # noqa: F401,F403
