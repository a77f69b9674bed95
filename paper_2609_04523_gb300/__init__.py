"""GB300 (sm_103a) fused attention: forward and backward passes (causal /
non-causal, grouped-query heads, packed variable-length sequences), a
paged-cache decode step and a latent (MLA) decode step.

The compute path is the CUDA library built from csrc/ (C ABI in
include/mk_attn.h); ``binding`` marshals arguments to it.  Importing this
package does not load the library; the first call does, and raises if it is
missing."""
from .binding import (MkAttnError, attn_bwd, attn_fwd, decode_paged, library_path, load_library,
                      mla_decode_paged,
                      mk_attn_bwd, mk_attn_bwd_workspace_bytes, mk_attn_check_status,
                      mk_attn_decode_paged, mk_attn_decode_workspace_bytes, mk_attn_error_string,
                      mk_attn_fwd, mk_attn_version)

__all__ = ["MkAttnError", "attn_bwd", "attn_fwd", "decode_paged", "library_path", "load_library",
           "mla_decode_paged",
           "mk_attn_bwd", "mk_attn_bwd_workspace_bytes", "mk_attn_check_status",
           "mk_attn_decode_paged", "mk_attn_decode_workspace_bytes", "mk_attn_error_string",
           "mk_attn_fwd", "mk_attn_version"]
