"""GB300 (sm_103a) implementation of TADM's anchor-cache reverse-diffusion sampling loop.

The compute path lives in ``csrc/`` (CUDA kernels + the C ABI of
``include/tadm.h``, built into ``_lib/libtadm.so``); ``tadm`` is the thin
ctypes binding.
"""
from .tadm import (TadmError, TadmModel, load_library, make_config, tadm_layer_cost, tadm_plan,  # noqa: F401
                   tadm_weight_inventory, upload_weights)
