"""GB300-native paged 4-bit KV attention (the KVExec hot path of JustFit).

The compute lives in libjfkv.so (hand-written sm_103a CUDA behind a C ABI,
include/jfkv.h); ``binding`` marshals torch tensors into those calls.
"""
from .binding import (  # noqa: F401
    KVPool, JfError, decode_workspace, default_num_splits, jf_attn_workspace_bytes,
    jf_kv_checkpoint, jf_kv_page_bytes, jf_kv_quantize_append, jf_kv_restore,
    jf_paged_decode_append_attn, jf_paged_decode_attn, jf_paged_decode_attn_noalloc,
    jf_paged_verify_attn, jf_prefill_chunk_attn, jf_prefill_workspace_bytes, lib,
    status_string, version, verify_workspace, default_verify_splits, workspace_status,
    JF_FMT_AFFINE4_G64, JF_FMT_TQ4, Tq4Codec, jf_kv_page_bytes_fmt, jf_tq4_codebook,
    jf_prefill_batch_attn, jf_reservation_pages, prefill_batch_workspace, default_prefill_splits,
    jf_prefill_chunk_workspace_bytes, prefill_chunk_workspace,
)
