"""GB300-native hot path of Looped Latent Attention (LLA): the cross-loop KV codec and the
attention that reads its latents, as a C-ABI CUDA library (include/lla.h, liblla.so) with a
thin Python binding (``lla``) and seeded synthetic workloads (``workloads``)."""
from . import workloads  # noqa: F401  (pure Python; the CUDA library loads on first call)

__all__ = ["lla", "workloads", "build"]
