"""GB300-native true-tail incremental memory maintenance (sm_103a CUDA kernels
behind a C ABI, include/kvm.h).  `kvm.Context` is the Python binding."""
from . import kvm  # noqa: F401
from .kvm import Context, KvmError, load_library, LAYER_ATTN, LAYER_GDN  # noqa: F401
