"""CPU oracle (fp64) for the split-head vocabulary projection.

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and
bench.py's cpu_baseline / reference leg, never by the product path.
"""
from .sph_oracle import *  # noqa: F401,F403
from .sph_oracle import (decode_bf16, decode_e4m3, round_fp32_to_bf16,  # noqa: F401
                         philox4x32_10, philox_uniform, gathered_matvec,
                         quantize_rows, payload_bytes, partial_logits,
                         local_partial, fuse, softmax_rows, inverse_cdf,
                         sample_rows, fuse_sample, verify_core,
                         compact_index, verify_draft, E4M3_VALUES, draw,
                         chunk_bounds, quantize_chunks, payload_bytes_chunked,
                         fuse_chunks, split_step)
