"""GB300 (sm_103a) KV-PRM verify-token scoring: a C-ABI CUDA library
(include/kvprm.h, csrc/) and its ctypes binding (kvprm.py)."""
from .kvprm import (KvprmConfig, KvprmError, KvprmLora, KvprmWeights, Scorer, kvprm_plan_projection, kvprm_set_lora, kvprm_set_readout_depth, kvprm_attention, kvprm_attention_noalloc, kvprm_check_device,  # noqa: F401
                    kvprm_create, kvprm_debug_attn_out, kvprm_debug_hidden, kvprm_debug_layers, kvprm_projection, kvprm_destroy, kvprm_get_profile, kvprm_resolve,
                    kvprm_score, kvprm_score_async, kvprm_score_host, kvprm_set_debug, kvprm_set_profile, kvprm_set_trace, kvprm_get_trace, kvprm_get_trace_events, lib,
                    library_path)
