"""GB300-native (sm_103a) hot path of LoGo's token-level local/global attention.

The computation lives in a C-ABI CUDA library (``include/logo.h``,
``csrc/*.cu``); ``logo`` is its thin Python binding and ``layer`` chains the
entry points into one forward/backward step of the attention layer.
"""
from .logo import (LOGO_SELECT_RATIO, LOGO_SELECT_THRESHOLD, LogoError, logo_combine, logo_combine_bwd,  # noqa: F401
                   logo_get_device_status, logo_global_sparse_attn_bwd, logo_global_sparse_attn_fwd,
                   logo_local_attn_bwd, logo_local_attn_fwd, logo_num_sms, logo_select)
