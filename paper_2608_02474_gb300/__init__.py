"""EchoCache cached DiT step on GB300 (sm_103a): C-ABI library + thin binding."""
from . import echocache  # noqa: F401
from .echocache import (BlockDims, DeviceBlock, EchoError, echo_attention, echo_audio_energy,  # noqa: F401
                        echo_block_step, echo_cache_dequant, echo_cache_quant,
                        echo_get_device_error, echo_layernorm, echo_linear,
                        echo_precompute_cross_kv, echo_select, echo_select_workspace_size,
                        echo_workspace_size, lib)
