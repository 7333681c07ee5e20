"""EchoCache cached DiT step on GB300 (sm_103a): C-ABI library + thin binding."""
from . import echocache  # noqa: F401
from .echocache import (CACHE_BF16, CACHE_INT8, CACHE_REF, BlockDims, DeviceBlock,  # noqa: F401
                        DeviceCache, EchoError, echo_attention, echo_audio_energy,
                        echo_block_step, echo_block_step_cache, echo_cache_dequant,
                        echo_cache_quant, echo_get_device_error, echo_layernorm, echo_linear,
                        echo_precompute_cross_kv, echo_select, echo_select_cache,
                        echo_select_random, echo_select_uniform, echo_select_workspace_size,
                        echo_step_delta, echo_update_rate, echo_workspace_size, lib)
