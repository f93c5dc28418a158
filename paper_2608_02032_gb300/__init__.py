"""GB300-native (sm_103a) hot path of DART, "Decoded Attention over Recurrent
sTates" (arXiv 2608.02032): the chunked SSD scan with chunk state memories,
state-memory attention with the gated merge, and the decode step over the
chunk-memory cache, as hand-written CUDA kernels behind the C ABI in
``include/dart.h``.

``binding`` exposes the C entry points under their own names; ``api``
allocates outputs with PyTorch and calls them; ``workloads`` draws the
seeded synthetic inputs. Nothing here computes on the CPU.
"""
from .binding import (DartError, dart_chunk_scan, dart_decode_step, dart_get_device_status,  # noqa: F401
                      dart_launch_count,
                      dart_sma_forward, dart_workspace_size, make_dims)
