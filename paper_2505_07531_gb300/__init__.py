"""GB300-native per-group 3/4-bit weight quantization fused into matmul.

The compute path is the CUDA library ``lib/libqx.so`` (sources in ``csrc/``,
C ABI in ``include/qx.h``); :mod:`.qx` is its thin ctypes binding.
"""
from .qx import (  # noqa: F401
    F16,
    F32,
    GEMV_PDL,
    LUT,
    UNIFORM,
    PackedMatrix,
    QxError,
    Recipe,
    dequant,
    device_status,
    gemm,
    gemv,
    gemv_multi,
    library_path,
    packed_size,
    quantize,
    version,
)
