"""GB300-native slot attention for Zarya's slotted speculative decoding.

The hot path of Mode B (Sec. 5.2): a block of S slots x L query tokens per
sequence attends over its cached prefix plus itself, block-bidirectionally
in the draft pass and causally in the verification pass, and the accepted
tokens are appended to the KV cache. The compute lives in ``libzarya.so``
(hand-written sm_103a CUDA behind the C ABI of ``include/zarya.h``); this
package is its Python binding.
"""
from ._binding import (  # noqa: F401
    APPEND_COMMIT, APPEND_STAGE, BF16, FP32, MASK_BIDIR_BLOCK, MASK_SLOT_CAUSAL, AttnDesc,
    ZaryaError, check_device_error, header_functions, kv_append, load, make_desc, slot_attn,
    status_string, version, workspace_size)
