"""CertKV exact-budget KV-cache compression and packed decode for GB300.

The compute path is the CUDA library built from ``csrc/`` (sm_103a) behind the
C ABI of ``include/certkv.h``; ``certkv`` is its thin Python binding and
``workloads`` draws the seeded synthetic inputs.
"""
from .certkv import (CertKVError, Packed, certkv_compress, certkv_compress_scored,  # noqa: F401
                     certkv_curves, certkv_decode_attn, certkv_decode_workspace_bytes,
                     certkv_default_params, certkv_live_budget, certkv_read_status,
                     certkv_score, certkv_strerror, certkv_workspace_bytes, load_library)
