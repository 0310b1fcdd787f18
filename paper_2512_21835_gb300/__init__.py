"""GB300-native LOIP hot path: lossless LLaMA-style decoding with layer weights
streamed from pinned host memory into device slots (arXiv 2512.21835, one GPU).

The compute runs in libloip.so (CUDA, sm_103a); `loip` is its Python binding.
"""
from . import configs, inputs  # noqa: F401

__all__ = ["configs", "inputs", "loip"]
