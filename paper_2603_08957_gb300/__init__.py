"""GB300 executor for upper-case-lower-case EinSum over tensor-relations.

The compute lives in ``libucl.so`` (hand-written sm_103a CUDA behind the C ABI
of ``include/ucl.h``); ``Context`` / ``Relation`` are its Python binding.
"""
from .ucl import BF16, F32, Context, Relation, UclError, plan, plan_dag  # noqa: F401
