"""GB300-native multipoint post-training quantization (arXiv 2002.09049).

The compute path lives in the C-ABI library ``libmpq.so`` (hand-written CUDA for sm_103a, built
from ``csrc/``); ``binding`` marshals torch tensors into its entry points and loads the library
on first use.  There is no CPU fallback: calling an entry point without the compiled library
raises.
"""
from . import overhead, workloads  # noqa: F401
from .binding import (MPQ_ALLOC_BUDGET, MPQ_ALLOC_THRESHOLD, MPQ_CENTER_PER_CHANNEL,  # noqa: F401
                      MPQ_CENTER_PER_LAYER, MPQ_CLIP_PER_CHANNEL, MPQ_CLIP_PER_LAYER, MPQError,
                      PackedLayout, mpq_allocate_points, mpq_center_weights, mpq_clip_search,
                      mpq_multipoint_linear, mpq_output_error, mpq_output_error_noalloc,
                      mpq_pack_layout, mpq_pack_points, mpq_quantize_layer,
                      mpq_quantize_layer_adaptive, mpq_reconstruct,
                      mpq_status_string, mpq_version)
