"""GB300-native (sm_103a) QUASAR per-step loss-aware reconstruction.

The product is the C-ABI CUDA library ``_build/libquasar.so`` (declared in
``include/quasar.h``); ``quasar`` is its thin ctypes binding, ``api``
allocates outputs with PyTorch, ``workloads`` draws seeded synthetic inputs.
"""
from .quasar import (QuasarError, QuasarStatus, quasar_debug_force_timeout,  # noqa: F401
                     quasar_debug_set_stats, quasar_get_device_status, quasar_recon_int,
                     quasar_recon_nvfp4, quasar_status_string, quasar_tensor_amax,
                     quasar_version)
