"""ctypes binding of libsky_slice.so: the C ABI of include/sky_slice.h and
include/sky_ops.h under the same names.

The binding only marshals arguments (pointers, sizes, enums); every step of
the encoder slice runs in the library's CUDA kernels.  Loading fails loudly
when the library has not been built: there is no fallback implementation.
"""
from __future__ import annotations

import ctypes as C
import os

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libsky_slice.so")

SKY_OK, SKY_ERR_INVALID_ARG, SKY_ERR_OOM, SKY_ERR_CUDA, SKY_ERR_STATE, SKY_ERR_TIMEOUT, \
    SKY_ERR_UNSUPPORTED, SKY_ERR_INFEASIBLE = range(8)
SKY_DTYPE_BF16, SKY_DTYPE_FP32 = 0, 1
SKY_GEMM_XWT, SKY_GEMM_XW, SKY_GEMM_XTW = 0, 1, 2
SKY_EPI_STORE, SKY_EPI_BIAS_GELU, SKY_EPI_GELU_BWD = 0, 1, 2
SKY_NUM_PARAMS = 12


class SkySliceConfig(C.Structure):
    _fields_ = [("width", C.c_int32), ("heads", C.c_int32), ("ffn", C.c_int32),
                ("layer_begin", C.c_int32), ("layer_end", C.c_int32),
                ("max_batch", C.c_int32), ("max_seq", C.c_int32),
                ("dtype", C.c_int), ("ln_eps", C.c_float), ("io_fp32", C.c_int32),
                ("stash_slots", C.c_int32)]


class SkyLayerCost(C.Structure):
    _fields_ = [("layer", C.c_int32), ("_pad", C.c_int32),
                ("fwd_ms", C.c_double), ("bwd_ms", C.c_double),
                ("fwd_flops", C.c_double), ("bwd_flops", C.c_double),
                ("param_bytes", C.c_uint64), ("grad_bytes", C.c_uint64),
                ("stash_bytes", C.c_uint64), ("workspace_bytes", C.c_uint64)]


class SkyKernelStat(C.Structure):
    _fields_ = [("name", C.c_char * 32), ("launches", C.c_int64), ("total_ms", C.c_double),
                ("flops", C.c_double), ("bytes", C.c_double)]


class SkyError(RuntimeError):
    def __init__(self, status: int, where: str, message: str):
        super().__init__(f"{where}: status {status} ({STATUS_NAMES.get(status, '?')}): {message}")
        self.status = status


STATUS_NAMES = {SKY_OK: "SKY_OK", SKY_ERR_INVALID_ARG: "SKY_ERR_INVALID_ARG",
                SKY_ERR_OOM: "SKY_ERR_OOM", SKY_ERR_CUDA: "SKY_ERR_CUDA",
                SKY_ERR_STATE: "SKY_ERR_STATE", SKY_ERR_TIMEOUT: "SKY_ERR_TIMEOUT",
                SKY_ERR_UNSUPPORTED: "SKY_ERR_UNSUPPORTED", SKY_ERR_INFEASIBLE: "SKY_ERR_INFEASIBLE"}

class SkyAllocProblem(C.Structure):
    _fields_ = [("devices", C.c_int32), ("layers", C.c_int32),
                ("dt", C.POINTER(C.c_double)), ("dm", C.POINTER(C.c_double)),
                ("ct", C.POINTER(C.c_double)), ("lf", C.POINTER(C.c_double)),
                ("lm", C.POINTER(C.c_double))]


SKY_COST_CT_PER_DEVICE, SKY_COST_CT_PER_LAYER = 0, 1
SKY_OPT_SGD, SKY_OPT_ADAMW = 0, 1


class SkyOptimizerConfig(C.Structure):
    _fields_ = [("kind", C.c_int32), ("lr", C.c_float), ("beta1", C.c_float),
                ("beta2", C.c_float), ("eps", C.c_float), ("weight_decay", C.c_float),
                ("momentum", C.c_float)]

_VP, _I32, _SZ = C.c_void_p, C.c_int32, C.c_size_t
_SIGNATURES = {
    "sky_slice_create": (C.c_int, [C.POINTER(SkySliceConfig), C.POINTER(_VP)]),
    "sky_slice_destroy": (C.c_int, [_VP]),
    "sky_slice_set_params": (C.c_int, [_VP, _I32, C.POINTER(_VP), C.c_int]),
    "sky_slice_get_params": (C.c_int, [_VP, _I32, C.POINTER(_VP), C.c_int]),
    "sky_slice_get_grads": (C.c_int, [_VP, _I32, C.POINTER(_VP), C.c_int]),
    "sky_slice_forward": (C.c_int, [_VP, _VP, _VP, _I32, _I32, _VP, _VP]),
    "sky_slice_backward": (C.c_int, [_VP, _VP, _VP, _VP]),
    "sky_slice_forward_slot": (C.c_int, [_VP, _VP, _VP, _I32, _I32, _VP, _I32, _VP]),
    "sky_slice_backward_slot": (C.c_int, [_VP, _VP, _VP, _I32, _I32, _VP]),
    "sky_device_delay": (C.c_int, [C.c_uint64, _VP]),
    "sky_slice_step_graph_create": (C.c_int, [_VP, _VP, _VP, _I32, _I32, _VP, _VP, _VP, _VP]),
    "sky_slice_step_graph_launch": (C.c_int, [_VP, _VP]),
    "sky_slice_layer_cost": (C.c_int, [_VP, _I32, _I32, C.POINTER(_I32), _I32,
                                        C.POINTER(SkyLayerCost), _I32]),
    "sky_slice_sync": (C.c_int, [_VP]),
    "sky_slice_set_profiling": (C.c_int, [_VP, C.c_int]),
    "sky_slice_kernel_stats": (C.c_int, [_VP, C.POINTER(SkyKernelStat), _I32, C.POINTER(_I32)]),
    "sky_slice_memory": (C.c_int, [_VP] + [C.POINTER(C.c_uint64)] * 4),
    "sky_debug_set_alloc_cap": (None, [C.c_uint64]),
    "sky_launch_count": (C.c_int64, []),
    "sky_status_string": (C.c_char_p, [C.c_int]),
    "sky_last_error": (C.c_char_p, []),
    "sky_gemm_workspace_bytes": (_SZ, [C.c_int, _I32, _I32, _I32, C.c_int, C.c_int]),
    "sky_gemm": (C.c_int, [C.c_int, _I32, _I32, _I32, C.c_int, _VP, _VP, _VP, C.c_int, C.c_int,
                           _VP, _VP, _VP, _VP, _SZ, _VP, _VP]),
    "sky_attention_fwd": (C.c_int, [_VP, _VP, _I32, _I32, _I32, _I32, C.c_int, _VP, _VP, _VP,
                                    _VP]),
    "sky_attention_bwd_workspace_bytes": (_SZ, [_I32, _I32, _I32, _I32]),
    "sky_attention_bwd": (C.c_int, [_VP, _VP, _VP, _VP, _VP, _I32, _I32, _I32, _I32, C.c_int,
                                    _VP, _VP, _SZ, _VP, _VP]),
    "sky_layernorm_fwd": (C.c_int, [_VP, _VP, _VP, _VP, _I32, _I32, C.c_float, C.c_int, _VP,
                                    _VP, _VP, _VP, _VP, _VP]),
    "sky_layernorm_bwd_workspace_bytes": (_SZ, [_I32, _I32]),
    "sky_layernorm_bwd": (C.c_int, [_VP, C.c_int, _VP, _VP, _VP, _VP, _VP, _I32, _I32, C.c_int,
                                    _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP]),
    "sky_add_f32": (C.c_int, [_VP, _VP, C.c_int64, C.c_int, _VP, _VP]),
    "sky_to_f32": (C.c_int, [_VP, C.c_int64, C.c_int, _VP, _VP]),
    "sky_bias_gelu_fwd": (C.c_int, [_VP, _VP, _I32, _I32, C.c_int, _VP, _VP, _VP]),
    "sky_gelu_bwd": (C.c_int, [_VP, _VP, _I32, _I32, C.c_int, _VP, _VP]),
    "sky_column_sum_workspace_bytes": (_SZ, [_I32, _I32]),
    "sky_column_sum": (C.c_int, [_VP, _I32, _I32, C.c_int, _VP, _VP, _SZ, _VP]),
    "sky_column_sum_noalloc": (C.c_int, [_VP, _I32, _I32, C.c_int, _VP, _VP]),
    "sky_debug_gemm_fault": (None, [C.c_uint64, C.c_int32]),
    "sky_device_sm_count": (_I32, []),
    "sky_slice_optimizer_init": (C.c_int, [_VP, C.POINTER(SkyOptimizerConfig)]),
    "sky_slice_optimizer_step": (C.c_int, [_VP, C.c_float, _VP]),
    "sky_slice_get_optimizer_state": (C.c_int, [_VP, _I32, _I32, C.POINTER(_VP)]),
    "sky_alloc_even": (C.c_int, [_I32, _I32, C.POINTER(_I32)]),
    "sky_alloc_coarse": (C.c_int, [C.POINTER(SkyAllocProblem), C.POINTER(_I32)]),
    "sky_alloc_finetune": (C.c_int, [C.POINTER(SkyAllocProblem), _I32, C.POINTER(_I32),
                                     C.POINTER(_I32)]),
    "sky_alloc_heuristic": (C.c_int, [C.POINTER(SkyAllocProblem), _I32, C.POINTER(_I32)]),
    "sky_alloc_workloads": (C.c_int, [C.POINTER(SkyAllocProblem), C.POINTER(_I32), C.c_int,
                                      C.POINTER(C.c_double)]),
    "sky_alloc_best_ordered": (C.c_int, [C.POINTER(SkyAllocProblem), C.POINTER(_I32),
                                         C.POINTER(C.c_double)]),
    "sky_alloc_milp_exact": (C.c_int, [C.POINTER(SkyAllocProblem), C.POINTER(_I32),
                                       C.POINTER(C.c_double)]),
}

_lib = None


def lib() -> C.CDLL:
    """Loads libsky_slice.so (built by ``paper_2202_11836_gb300.build``)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"{LIB_PATH} is missing: build it with `python -m paper_2202_11836_gb300.build` "
                "(or __graft_entry__.build()); there is no non-CUDA fallback")
        l = C.CDLL(LIB_PATH)
        for name, (res, args) in _SIGNATURES.items():
            fn = getattr(l, name)
            fn.restype = res
            fn.argtypes = args
        _lib = l
    return _lib


def last_error() -> str:
    return lib().sky_last_error().decode()


def check(status: int, where: str) -> None:
    if status != SKY_OK:
        raise SkyError(status, where, last_error())


def call(name: str, *args) -> None:
    """Calls an ABI function and raises SkyError on a non-OK status."""
    check(getattr(lib(), name)(*args), name)
