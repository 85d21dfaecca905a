"""GB300-native (sm_103a) verify/arbitrate round of collaborative speculative
decoding (CoSpec): paged verify attention, a tcgen05 LM head fused with
argmax and log-prob statistics, mismatch arbitration and accept/commit, all
behind the C ABI of include/cospec.h (libcospec.so)."""
from . import cospec, workload  # noqa: F401

__all__ = ["cospec", "workload"]
