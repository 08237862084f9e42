"""GB300-native Hierarchical Sparse Attention (HSA) hot path.

All compute is hand-written CUDA for sm_103a in libhsa.so (C ABI in
include/hsa.h); this package only builds it and marshals torch tensors into
its calls.
"""
from .binding import (  # noqa: F401
    CHUNK,
    HSA_OP_BACKWARD,
    HSA_OP_BACKWARD_ATTENTION,
    HSA_OP_SELECT_BACKWARD,
    HSA_OP_FORWARD,
    HSA_OP_INDEX,
    HSA_OP_SELECT,
    DecodeShape,
    HsaError,
    Shape,
    Workspaces,
    backward,
    backward_attention,
    select_backward,
    build_index,
    chunk_pool,
    decode,
    decode_index,
    decode_indexed,
    decode_noalloc,
    memory_append,
    decode_workspace_size,
    check,
    new_workspace,
    status_bytes,
    selftest_score_tile,
    selftest_wait_timeout,
    forward,
    hsa_backward_path,
    hsa_forward_path,
    kernel_launches,
    lib_path,
    load,
    select_topk,
    status_string,
    workspace_size,
)
from .build import build  # noqa: F401

__version__ = "0.1.0"
