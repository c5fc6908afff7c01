"""GB300 (sm_103a) three-stage attention: prefill, prefill_kv and decode.

The compute path is the C-ABI library ``libattn_gb300.so`` (include/attn.h) with
hand-written CUDA kernels; ``attention.Attention`` is a thin torch-facing wrapper.
Importing this package loads nothing; ``attention`` loads the library on use.
"""
__all__ = ["attention", "build"]
