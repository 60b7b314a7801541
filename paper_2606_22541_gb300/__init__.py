"""GB300-native expert-side MoE layer of ASAP's data-parallel prefill path.

The layer (top-k gating, per-expert counts and offsets, dispatch, tcgen05
grouped SwiGLU expert FFN with a shared expert, weighted combine) lives in
libasap_moe.so (C ABI in include/asap_moe.h); ``api`` is its Python binding.
Importing this package does not load the library; the first API call does,
and fails loudly when it has not been built.
"""
__all__ = ["api", "configs", "inputs", "build"]
