"""LoopGuard decode path on GB300 (sm_103a): decode attention fused with the guard's per-head
statistics, the online loop-onset test, and the pruning / in-place compaction of the KV cache
under a fixed budget, plus the H2O eviction comparator.  The compute runs in liblg.so (CUDA,
C ABI in include/lg.h); ``lg`` is its Python binding."""
from . import lg  # noqa: F401
