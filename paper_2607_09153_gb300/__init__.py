"""GB300 (sm_103a) KV-PRM verify-token scoring: a C-ABI CUDA library
(include/kvprm.h, csrc/) and its ctypes binding (kvprm.py)."""
from .kvprm import (KVPRM_EINVAL, KVPRM_ECAPACITY, KVPRM_ECUDA, KVPRM_EINDEX, KVPRM_ENOMEM, KVPRM_ETIMEOUT,  # noqa: F401
                    KVPRM_EUNSUPPORTED, KVPRM_OK, KVPRM_PLAN_FUSE, KvprmConfig, kvprm_plan_attention, KvprmError, KvprmLora, KvprmWeights, Scorer, kvprm_plan_projection, kvprm_set_lora, kvprm_set_readout_depth, kvprm_attention, kvprm_attention_noalloc, kvprm_check_device,  # noqa: F401
                    kvprm_debug_inject_error, kvprm_debug_set_alloc_limit, kvprm_debug_wait_probe,
                    kvprm_create, kvprm_debug_attn_out, kvprm_debug_hidden, kvprm_debug_layers, kvprm_projection, kvprm_destroy, kvprm_get_profile, kvprm_resolve,
                    kvprm_score, kvprm_score_async, kvprm_score_host, kvprm_score_grad, kvprm_steer, kvprm_set_debug, kvprm_set_profile, kvprm_set_trace, kvprm_get_trace, kvprm_get_trace_events, lib,
                    library_path)
