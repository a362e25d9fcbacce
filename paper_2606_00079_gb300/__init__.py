"""Python binding of libbitsmoe, the GB300 BitsMoE quantized MoE-layer forward.

Argument marshalling only: every step of the forward runs in the library's
CUDA kernels.  The functions carry the C ABI's names (see include/bitsmoe.h);
PyTorch is used only for device memory and streams by the convenience wrapper
``moe_forward``.  There is no CPU fallback: if the compiled library is missing
every entry point raises ``BitsMoEUnavailable``.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libbitsmoe.so")

OK = 0
ERR = {
    -1: "INVALID_ARG", -2: "SHAPE", -3: "UNSUPPORTED_BITS", -4: "WORKSPACE_TOO_SMALL",
    -5: "ALIGNMENT", -6: "CUDA", -7: "OOM", -8: "TIMEOUT", -9: "DEVICE_BOUNDS", -10: "BLOB",
    -11: "WORKSPACE_STATE",
}
ERR_CODE = {v: k for k, v in ERR.items()}

# Every C entry point declared in include/bitsmoe.h, with (restype, argtypes).
_P = ctypes.c_void_p
_I = ctypes.c_int
_SZ = ctypes.c_size_t


class _LayerHost(ctypes.Structure):
    _fields_ = [("D", ctypes.c_int32), ("E", ctypes.c_int32), ("I", ctypes.c_int32),
                ("n", ctypes.c_int32), ("group", ctypes.c_int32),
                ("basis", _P * 3), ("bits", _P), ("alpha", _P), ("codes", _P),
                ("scale", _P), ("zero", _P)]


class _Bytes(ctypes.Structure):
    _fields_ = [("total", ctypes.c_uint64), ("basis", ctypes.c_uint64),
                ("codes_padded", ctypes.c_uint64), ("meta", ctypes.c_uint64)]


SIGNATURES = {
    "bitsmoe_pack": (_I, [ctypes.POINTER(_LayerHost), _I, ctypes.POINTER(_P)]),
    "bitsmoe_pack_to_host": (_I, [ctypes.POINTER(_LayerHost), ctypes.POINTER(_P), ctypes.POINTER(_SZ)]),
    "bitsmoe_blob_free": (None, [_P]),
    "bitsmoe_load_blob": (_I, [_P, _SZ, _I, ctypes.POINTER(_P)]),
    "bitsmoe_unpack_blob": (_I, [_P, _SZ, ctypes.POINTER(_LayerHost)]),
    "bitsmoe_unpack": (_I, [_P, ctypes.POINTER(_LayerHost)]),
    "bitsmoe_layer_dims": (_I, [_P, ctypes.POINTER(ctypes.c_int32)]),
    "bitsmoe_layer_bytes": (_I, [_P, ctypes.POINTER(_Bytes)]),
    "bitsmoe_expert_moved_bytes": (_I, [_P, _I, ctypes.POINTER(ctypes.c_uint64)]),
    "bitsmoe_profile_forward": (_I, [_P, _P, _I, _I, _P, _P, _P, _SZ, _P, ctypes.POINTER(ctypes.c_float)]),
    "bitsmoe_workspace_bytes": (_SZ, [_P, _I, _I]),
    "bitsmoe_forward_launches": (_I, [_P, _I, _I]),
    "bitsmoe_block_forward_launches": (_I, [_P, _I, _I]),
    "bitsmoe_forward_plan": (_I, [_P, _I, _I]),
    "bitsmoe_moe_forward": (_I, [_P, _P, _I, _I, _P, _P, _P, _SZ, _P]),
    "bitsmoe_moe_forward_host": (_I, [_P, _P, _I, _I, _P, _P, _P, _SZ, _P]),
    "bitsmoe_moe_forward_host_async": (_I, [_P, _P, _I, _I, _P, _P, _P, _SZ, _P]),
    "bitsmoe_moe_forward_noalloc": (_I, [_P, _P, _I, _I, _P, _P, _P]),
    "bitsmoe_noalloc_last_status": (_I, [_P]),
    "bitsmoe_rmsnorm_router": (_I, [_P, _P, ctypes.c_float, _I, _I, _I, _P, _P, _P]),
    "bitsmoe_moe_block_forward": (_I, [_P, _P, ctypes.c_float, _I, _I, _P, _P, _SZ, _P]),
    "bitsmoe_quantize_units": (_I, [_P, _P, ctypes.c_int64, _I, _I, _I, _P, _P, _P, _P, _P]),
    "bitsmoe_allocate_workspace_bytes": (_SZ, [ctypes.c_int64]),
    "bitsmoe_projection_budget": (_I, [ctypes.c_int64] * 5 + [ctypes.POINTER(ctypes.c_int64)]),
    "bitsmoe_allocate_bits": (_I, [_P, _P, _P, ctypes.c_float, ctypes.c_int64, _I, ctypes.POINTER(ctypes.c_float),
                                   ctypes.c_int64, _P, _P, _SZ, _P]),
    "bitsmoe_profile_allocate_bits": (_I, [_P, _P, _P, ctypes.c_float, ctypes.c_int64, _I,
                                           ctypes.POINTER(ctypes.c_float), ctypes.c_int64, _P, _P, _SZ, _P,
                                           ctypes.POINTER(ctypes.c_float)]),
    "bitsmoe_importance_workspace_bytes": (_SZ, [ctypes.c_int64, _I, _I, _I, _I]),
    "bitsmoe_importance": (_I, [_P, _P, ctypes.c_int64, _I, _I, _I, _I, _I, ctypes.POINTER(_P), ctypes.POINTER(_P),
                                ctypes.POINTER(_P), _P, _P, _SZ, _P]),
    "bitsmoe_decompose_workspace_bytes": (_SZ, [_I, _I, _I, _I]),
    "bitsmoe_shared_basis": (_I, [_I, _P, _I, _I, _I, _P, _P, _P, _P, _P, _SZ, _I, _P, _P, _P]),
    "bitsmoe_calibration_gram": (_I, [_P, _P, ctypes.c_int64, _I, _P, _P]),
    "bitsmoe_block_norm_outputs": (_I, [_P, _I, _I, ctypes.POINTER(_SZ), ctypes.POINTER(_SZ)]),
    "bitsmoe_last_device_status": (_I, [_P, _P]),
    "bitsmoe_free": (None, [_P]),
    "bitsmoe_strerror": (ctypes.c_char_p, [_I]),
    "bitsmoe_last_cuda_error": (_I, []),
    "bitsmoe_debug_wait_limit": (_I, [_I, ctypes.c_longlong]),
    "bitsmoe_debug_single_token_kernel": (_I, [_I]),
    "bitsmoe_debug_bounds": (_I, [_I]),
    "bitsmoe_debug_shift_expert_records": (_I, [_P, _I, ctypes.c_longlong]),
}


class BitsMoEUnavailable(RuntimeError):
    pass


class BitsMoEError(RuntimeError):
    def __init__(self, code: int, where: str = ""):
        self.code = code
        name = ERR.get(code, str(code))
        extra = ""
        if code == -6:
            extra = f" (cudaError {_lib().bitsmoe_last_cuda_error()})"
        super().__init__(f"{where}: BITSMOE_ERR_{name}{extra}")


_lib_handle = None


def _lib():
    global _lib_handle
    if _lib_handle is None:
        if not os.path.exists(LIB_PATH):
            raise BitsMoEUnavailable(
                f"{LIB_PATH} is not built; build it with __graft_entry__.build() "
                "(the BitsMoE forward has no CPU fallback)")
        lib = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(lib, name)
            f.restype = res
            f.argtypes = args
        _lib_handle = lib
    return _lib_handle


def library_path() -> str:
    _lib()
    return LIB_PATH


def _check(rc: int, where: str):
    if rc != OK:
        raise BitsMoEError(rc, where)


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _host_struct(layer: Dict):
    """ctypes view of a host layer dict (see synth.make_layer); returns (struct, keepalive)."""
    keep = {}
    for k, dt in (("bits", np.uint8), ("alpha", np.float32), ("codes", np.uint16),
                  ("scale", np.uint16), ("zero", np.uint16)):
        keep[k] = np.ascontiguousarray(layer[k], dtype=dt)
    bases = [np.ascontiguousarray(layer["basis"][h], dtype=np.uint16) for h in range(3)]
    s = _LayerHost(int(layer["D"]), int(layer["E"]), int(layer["I"]), int(layer["n"]), int(layer["group"]))
    s.basis = (_P * 3)(*[_ptr(b) for b in bases])
    for k in ("bits", "alpha", "codes", "scale", "zero"):
        setattr(s, k, _ptr(keep[k]))
    keep["bases"] = bases
    return s, keep


def _empty_host(dims) -> Dict:
    D, E, I, n, group = dims
    ng = I // group
    return dict(D=D, E=E, I=I, n=n, group=group,
                basis=np.zeros((3, D, n), np.uint16), bits=np.zeros((3, E, n), np.uint8),
                alpha=np.zeros((3, E, n), np.float32), codes=np.zeros((3, E, n, I), np.uint16),
                scale=np.zeros((3, E, n, ng), np.uint16), zero=np.zeros((3, E, n, ng), np.uint16))


def _out_struct(out: Dict):
    s = _LayerHost(out["D"], out["E"], out["I"], out["n"], out["group"])
    s.basis = (_P * 3)(*[_ptr(out["basis"][h]) for h in range(3)])
    for k in ("bits", "alpha", "codes", "scale", "zero"):
        setattr(s, k, _ptr(out[k]))
    return s


class Layer:
    """A packed, device-resident layer (owns the library handle)."""

    def __init__(self, handle: int):
        self.handle = handle
        dims = (ctypes.c_int32 * 5)()
        _check(_lib().bitsmoe_layer_dims(handle, dims), "bitsmoe_layer_dims")
        self.D, self.E, self.I, self.n, self.group = (int(v) for v in dims)

    def free(self):
        if self.handle:
            _lib().bitsmoe_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass

    def bytes(self) -> Dict[str, int]:
        b = _Bytes()
        _check(_lib().bitsmoe_layer_bytes(self.handle, ctypes.byref(b)), "bitsmoe_layer_bytes")
        return dict(total=b.total, basis=b.basis, codes_padded=b.codes_padded, meta=b.meta)

    def expert_moved_bytes(self, e: int):
        """Algorithmic bytes of expert e per projection (gate, up, down)."""
        v = (ctypes.c_uint64 * 3)()
        _check(_lib().bitsmoe_expert_moved_bytes(self.handle, e, v), "bitsmoe_expert_moved_bytes")
        return [int(a) for a in v]


# --------------------------------------------------------------------------
# C-ABI entry points
# --------------------------------------------------------------------------
def bitsmoe_pack(layer: Dict, device: int = 0) -> Layer:
    s, keep = _host_struct(layer)
    h = _P()
    _check(_lib().bitsmoe_pack(ctypes.byref(s), device, ctypes.byref(h)), "bitsmoe_pack")
    return Layer(h.value)


def bitsmoe_pack_to_host(layer: Dict) -> np.ndarray:
    s, keep = _host_struct(layer)
    blob, nbytes = _P(), _SZ()
    _check(_lib().bitsmoe_pack_to_host(ctypes.byref(s), ctypes.byref(blob), ctypes.byref(nbytes)),
           "bitsmoe_pack_to_host")
    try:
        out = np.empty(nbytes.value, np.uint8)
        ctypes.memmove(_ptr(out), blob.value, nbytes.value)
    finally:
        _lib().bitsmoe_blob_free(blob)
    return out


def bitsmoe_load_blob(blob: np.ndarray, device: int = 0) -> Layer:
    blob = np.ascontiguousarray(blob, dtype=np.uint8)
    h = _P()
    _check(_lib().bitsmoe_load_blob(_ptr(blob), blob.nbytes, device, ctypes.byref(h)), "bitsmoe_load_blob")
    return Layer(h.value)


def bitsmoe_unpack_blob(blob: np.ndarray, dims) -> Dict:
    blob = np.ascontiguousarray(blob, dtype=np.uint8)
    out = _empty_host(dims)
    s = _out_struct(out)
    _check(_lib().bitsmoe_unpack_blob(_ptr(blob), blob.nbytes, ctypes.byref(s)), "bitsmoe_unpack_blob")
    return out


def bitsmoe_unpack(layer: Layer) -> Dict:
    out = _empty_host((layer.D, layer.E, layer.I, layer.n, layer.group))
    s = _out_struct(out)
    _check(_lib().bitsmoe_unpack(layer.handle, ctypes.byref(s)), "bitsmoe_unpack")
    return out


def bitsmoe_workspace_bytes(layer: Layer, T: int, top_k: int) -> int:
    return int(_lib().bitsmoe_workspace_bytes(layer.handle, T, top_k))


def bitsmoe_forward_launches(layer: Layer, T: int, top_k: int) -> int:
    """Kernels one forward call launches (1: the fused single-token kernel; 5: the chain)."""
    n = int(_lib().bitsmoe_forward_launches(layer.handle, T, top_k))
    if n < 0:
        raise BitsMoEError(n, "bitsmoe_forward_launches")
    return n


PLAN_FUSED, PLAN_DECODE_CHAIN, PLAN_TC_PROJECTIONS, PLAN_TC_GATE_UP, PLAN_TC_DOWN = 1, 2, 4, 8, 16
PLAN_CLUSTERED = 32


def bitsmoe_forward_plan(layer: Layer, T: int, top_k: int) -> int:
    """Bit set of how a T-token forward runs: PLAN_FUSED, PLAN_DECODE_CHAIN, PLAN_TC_PROJECTIONS,
    PLAN_TC_GATE_UP, PLAN_TC_DOWN, PLAN_CLUSTERED (with PLAN_FUSED: the clustered single-token kernel)."""
    n = int(_lib().bitsmoe_forward_plan(layer.handle, T, top_k))
    if n < 0:
        raise BitsMoEError(n, "bitsmoe_forward_plan")
    return n


def bitsmoe_block_forward_launches(layer: Layer, T: int, top_k: int) -> int:
    """Kernels one block forward launches (1: the fused kernel with its pre-norm; else norm/router + chain)."""
    n = int(_lib().bitsmoe_block_forward_launches(layer.handle, T, top_k))
    if n < 0:
        raise BitsMoEError(n, "bitsmoe_block_forward_launches")
    return n


def bitsmoe_moe_forward(x_ptr: int, logits_ptr: int, T: int, top_k: int, layer: Layer, y_ptr: int,
                        ws_ptr: int, ws_bytes: int, stream: int = 0) -> None:
    _check(_lib().bitsmoe_moe_forward(x_ptr, logits_ptr, T, top_k, layer.handle, y_ptr, ws_ptr,
                                      ws_bytes, stream), "bitsmoe_moe_forward")


def bitsmoe_moe_forward_host(x_bits: np.ndarray, logits: np.ndarray, top_k: int, layer: Layer,
                             ws_ptr: int, ws_bytes: int, stream: int = 0,
                             y_out: Optional[np.ndarray] = None) -> np.ndarray:
    """Forward from host arrays (x bf16 bits T x D, logits fp32 T x E) -> y fp32 T x D."""
    T = int(x_bits.shape[0])
    y = y_out if y_out is not None else np.empty((T, layer.D), np.float32)
    _check(_lib().bitsmoe_moe_forward_host(x_bits.ctypes.data, logits.ctypes.data, T, top_k, layer.handle,
                                           y.ctypes.data, ws_ptr, ws_bytes, stream), "bitsmoe_moe_forward_host")
    return y


NOALLOC_SCRATCH_BYTES = 8 << 20   # BITSMOE_NOALLOC_SCRATCH_BYTES


def bitsmoe_moe_forward_noalloc(x_ptr: int, logits_ptr: int, T: int, top_k: int, layer: Layer, y_ptr: int,
                                stream: int = 0) -> None:
    """The forward for callers that cannot allocate device memory: its scratch is
    the library's built-in array (NOALLOC_SCRATCH_BYTES per device, shared by all
    calls on that device, so overlapping calls race)."""
    _check(_lib().bitsmoe_moe_forward_noalloc(x_ptr, logits_ptr, T, top_k, layer.handle, y_ptr, stream),
           "bitsmoe_moe_forward_noalloc")


def bitsmoe_rmsnorm_router(h_ptr: int, w_router_ptr: int, eps: float, T: int, D: int, E: int,
                           x_out_ptr: int, logits_out_ptr: int, stream: int = 0) -> None:
    _check(_lib().bitsmoe_rmsnorm_router(h_ptr, w_router_ptr, eps, T, D, E, x_out_ptr, logits_out_ptr, stream),
           "bitsmoe_rmsnorm_router")


def bitsmoe_moe_block_forward(h_ptr: int, w_router_ptr: int, eps: float, T: int, top_k: int, layer: Layer,
                              ws_ptr: int, ws_bytes: int, stream: int = 0) -> None:
    _check(_lib().bitsmoe_moe_block_forward(h_ptr, w_router_ptr, eps, T, top_k, layer.handle, ws_ptr, ws_bytes,
                                            stream), "bitsmoe_moe_block_forward")


def bitsmoe_profile_forward(x_ptr: int, logits_ptr: int, T: int, top_k: int, layer: Layer, y_ptr: int,
                            ws_ptr: int, ws_bytes: int, stream: int = 0):
    """Forward with the five phases serialised and timed; returns their durations (ms)."""
    ms = (ctypes.c_float * 5)()
    _check(_lib().bitsmoe_profile_forward(x_ptr, logits_ptr, T, top_k, layer.handle, y_ptr, ws_ptr,
                                          ws_bytes, stream, ms), "bitsmoe_profile_forward")
    return [float(v) for v in ms]


def bitsmoe_quantize_units(p_ptr: int, bits_ptr: int, U: int, I: int, group: int, grid: int, codes_ptr: int,
                           scale_ptr: int, zero_ptr: int, status_ptr: int = 0, stream: int = 0) -> None:
    """Quantise U float units (device U x I fp32) into codes / fp16 scale / fp16 zero (device)."""
    _check(_lib().bitsmoe_quantize_units(p_ptr, bits_ptr, U, I, group, grid, codes_ptr, scale_ptr, zero_ptr,
                                         status_ptr, stream), "bitsmoe_quantize_units")


def bitsmoe_projection_budget(E: int, n: int, m: int, b_eq) -> int:
    """B_h = floor(E n b_eq - 16 n^2 / m) for b_eq given as a float, an int or a (num, den) pair."""
    from fractions import Fraction
    fr = Fraction(*b_eq) if isinstance(b_eq, tuple) else Fraction(str(b_eq))
    out = ctypes.c_int64()
    _check(_lib().bitsmoe_projection_budget(E, n, m, fr.numerator, fr.denominator, ctypes.byref(out)),
           "bitsmoe_projection_budget")
    return int(out.value)


def bitsmoe_allocate_workspace_bytes(U: int) -> int:
    return int(_lib().bitsmoe_allocate_workspace_bytes(U))


def bitsmoe_allocate_bits(p_ptr: int, alpha_ptr: int, beta_ptr: int, gamma: float, U: int, d: int, kappa,
                          budget: int, bits_ptr: int, ws_ptr: int, ws_bytes: int, stream: int = 0,
                          profile: bool = False):
    """Bit-width per unit (device, U bytes) for one projection type; with profile=True the call
    synchronises and returns the phase durations (ms: costs and hull, cut, fill)."""
    k = (ctypes.c_float * 3)(*[float(v) for v in kappa])
    if profile:
        ms = (ctypes.c_float * 3)()
        _check(_lib().bitsmoe_profile_allocate_bits(p_ptr, alpha_ptr, beta_ptr, gamma, U, d, k, budget, bits_ptr,
                                                    ws_ptr, ws_bytes, stream, ms), "bitsmoe_profile_allocate_bits")
        return [float(v) for v in ms]
    _check(_lib().bitsmoe_allocate_bits(p_ptr, alpha_ptr, beta_ptr, gamma, U, d, k, budget, bits_ptr, ws_ptr,
                                        ws_bytes, stream), "bitsmoe_allocate_bits")
    return None


def bitsmoe_last_device_status(ws_ptr: int, stream: int = 0) -> int:
    return int(_lib().bitsmoe_last_device_status(ws_ptr, stream))


def bitsmoe_block_norm_outputs(layer: Layer, T: int, top_k: int):
    """Byte offsets of a block forward's normalised x and router logits in its workspace."""
    xo, lo = _SZ(0), _SZ(0)
    _check(_lib().bitsmoe_block_norm_outputs(layer.handle, T, top_k, ctypes.byref(xo), ctypes.byref(lo)),
           "bitsmoe_block_norm_outputs")
    return int(xo.value), int(lo.value)


def bitsmoe_noalloc_last_status(stream: int = 0) -> int:
    """Device status of the no-allocation scratch on the current device (read and cleared)."""
    return int(_lib().bitsmoe_noalloc_last_status(stream))


def bitsmoe_strerror(code: int) -> str:
    return _lib().bitsmoe_strerror(code).decode()


# --------------------------------------------------------------------------
# torch convenience (device memory + streams only)
# --------------------------------------------------------------------------
class Workspace:
    """Device workspace sized for (T, top_k) on a layer, allocated (zero-filled) with torch."""

    def __init__(self, layer: Layer, T: int, top_k: int, device=None):
        import torch
        self.nbytes = bitsmoe_workspace_bytes(layer, T, top_k)
        if self.nbytes == 0:
            raise BitsMoEError(ERR_CODE["INVALID_ARG"], "bitsmoe_workspace_bytes")
        self.buf = torch.zeros(self.nbytes + 256, dtype=torch.uint8,
                               device=device if device is not None else f"cuda:{torch.cuda.current_device()}")
        base = self.buf.data_ptr()
        self.ptr = (base + 255) // 256 * 256


def moe_forward(layer: Layer, x_bits, logits, top_k: int, ws: Optional[Workspace] = None, y=None, stream=None):
    """y (fp32 T x D) = BitsMoE MoE-layer forward of x (int16/uint16 tensor of bf16 bits or a
    torch.bfloat16 tensor, T x D) with router logits (fp32 T x E), all on the device."""
    import torch
    T = int(x_bits.shape[0])
    if ws is None:
        ws = Workspace(layer, T, top_k, device=x_bits.device)
    if y is None:
        y = torch.empty((T, layer.D), dtype=torch.float32, device=x_bits.device)
    st = stream if stream is not None else torch.cuda.current_stream(x_bits.device)
    bitsmoe_moe_forward(x_bits.data_ptr(), logits.data_ptr(), T, top_k, layer, y.data_ptr(),
                        ws.ptr, ws.nbytes, st.cuda_stream)
    return y


def quantize_units(p, bits, group: int, grid: int = 256, stream=None):
    """Quantise the units in the rows of `p` (torch fp32 U x I on the device) with per-unit
    bit-widths `bits` (torch uint8, U) into the stored format; returns (codes uint16-as-int16
    U x I, scale, zero fp16 bit patterns U x I/group, status int32 tensor of one element)."""
    import torch
    U, I = int(p.shape[0]), int(p.shape[1])
    dev = p.device
    codes = torch.empty((U, I), dtype=torch.int16, device=dev)
    scale = torch.empty((U, I // group), dtype=torch.int16, device=dev)
    zero = torch.empty((U, I // group), dtype=torch.int16, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    st = stream if stream is not None else torch.cuda.current_stream(dev)
    bitsmoe_quantize_units(p.data_ptr(), bits.data_ptr(), U, I, group, grid, codes.data_ptr(), scale.data_ptr(),
                           zero.data_ptr(), status.data_ptr(), st.cuda_stream)
    return codes, scale, zero, status


def allocate_bits(p, alpha, beta, gamma: float, kappa, budget: int, stream=None):
    """Bit-widths (torch uint8, U) of the units in the rows of `p` (torch fp32 U x d on the
    device) with spectral energies `alpha` and importances `beta` (fp32, U) under `budget`."""
    import torch
    U, d = int(p.shape[0]), int(p.shape[1])
    dev = p.device
    bits = torch.empty(U, dtype=torch.uint8, device=dev)
    nb = bitsmoe_allocate_workspace_bytes(U)
    ws = torch.empty(nb + 256, dtype=torch.uint8, device=dev)
    st = stream if stream is not None else torch.cuda.current_stream(dev)
    bitsmoe_allocate_bits(p.data_ptr(), alpha.data_ptr(), beta.data_ptr(), gamma, U, d, kappa, budget,
                          bits.data_ptr(), (ws.data_ptr() + 255) // 256 * 256, nb, st.cuda_stream)
    ws.record_stream(st)   # the workspace is freed here but used by the kernels still queued on st
    return bits


def importance(x, logits, top_k: int, basis, alpha, factor, stream=None):
    """Importance beta (torch fp32, 3 x E x n) of every unit from calibration tokens: x (torch
    int16 bf16 bit patterns, T x D), logits (fp32, T x E), basis = (Phi_gate, Phi_up) fp32 D x n,
    alpha = (alpha_gate, alpha_up) fp32 E x n, factor = (P_gate, P_up, P_down) fp32 E x I x n,
    all on the device."""
    import torch
    T, D = int(x.shape[0]), int(x.shape[1])
    E = int(logits.shape[1])
    _, I, n = (int(v) for v in factor[0].shape)
    dev = x.device
    beta = torch.empty((3, E, n), dtype=torch.float32, device=dev)
    nb = int(_lib().bitsmoe_importance_workspace_bytes(T, E, I, n, top_k))
    ws = torch.empty(nb + 256, dtype=torch.uint8, device=dev)
    st = stream if stream is not None else torch.cuda.current_stream(dev)
    bp = (_P * 2)(*[b.data_ptr() for b in basis])
    ap = (_P * 2)(*[a.data_ptr() for a in alpha])
    fp = (_P * 3)(*[f.data_ptr() for f in factor])
    _check(_lib().bitsmoe_importance(x.data_ptr(), logits.data_ptr(), T, D, E, I, n, top_k, bp, ap, fp,
                                     beta.data_ptr(), (ws.data_ptr() + 255) // 256 * 256, nb, st.cuda_stream),
           "bitsmoe_importance")
    ws.record_stream(st)
    return beta


def shared_basis(W, side: str, max_sweeps: int = 30, stream=None):
    """Shared-basis decomposition of one projection type (torch fp32 on the device): side "in"
    takes W = E x d x D (gate/up, W_e = d x D), side "out" W = E x D x d (down, W_e = D x d).
    Returns (phi D x n, sigma n, alpha E x n, P E x n x d unit-major, sweeps, status) with
    n = min(D, E d); sweeps and status are device int tensors (one element each)."""
    import torch
    sd = {"in": 0, "out": 1}[side]
    E = int(W.shape[0])
    d, D = (int(W.shape[1]), int(W.shape[2])) if sd == 0 else (int(W.shape[2]), int(W.shape[1]))
    n = min(D, E * d)
    dev = W.device
    phi = torch.empty((D, n), dtype=torch.float32, device=dev)
    sigma = torch.empty((n,), dtype=torch.float32, device=dev)
    alpha = torch.empty((E, n), dtype=torch.float32, device=dev)
    P = torch.empty((E, n, d), dtype=torch.float32, device=dev)
    info = torch.zeros((2,), dtype=torch.int32, device=dev)   # sweeps, status
    nb = int(_lib().bitsmoe_decompose_workspace_bytes(sd, E, d, D))
    ws = torch.empty(nb + 256, dtype=torch.uint8, device=dev)
    st = stream if stream is not None else torch.cuda.current_stream(dev)
    _check(_lib().bitsmoe_shared_basis(sd, W.data_ptr(), E, d, D, phi.data_ptr(), sigma.data_ptr(), alpha.data_ptr(),
                                       P.data_ptr(), (ws.data_ptr() + 255) // 256 * 256, nb, max_sweeps,
                                       info.data_ptr(), info.data_ptr() + 4, st.cuda_stream),
           "bitsmoe_shared_basis")
    ws.record_stream(st)
    return phi, sigma, alpha, P, info[0:1], info[1:2]


def calibration_gram(x, g=None, stream=None):
    """H = sum_t g_t x_t x_t^T (torch fp32 D x D) from x (torch int16 bf16 bit patterns, T x D)
    and optional per-token weights g (fp32, T), on the device."""
    import torch
    T, D = int(x.shape[0]), int(x.shape[1])
    H = torch.empty((D, D), dtype=torch.float32, device=x.device)
    st = stream if stream is not None else torch.cuda.current_stream(x.device)
    _check(_lib().bitsmoe_calibration_gram(x.data_ptr(), g.data_ptr() if g is not None else None, T, D,
                                           H.data_ptr(), st.cuda_stream), "bitsmoe_calibration_gram")
    return H


def bitsmoe_debug_single_token_kernel(which: int) -> None:
    """Testing hook: 1 keeps single-token forwards on the fused kernel without clusters, 2 takes the
    clustered one wherever it fits, 0 restores the automatic choice."""
    _check(_lib().bitsmoe_debug_single_token_kernel(which), "bitsmoe_debug_single_token_kernel")


def bitsmoe_debug_bounds(on: int) -> None:
    """Testing hook: debug bounds checks of the single-token kernels' staging records (and a
    zero-filled slack after the image of layers packed while it is on)."""
    _check(_lib().bitsmoe_debug_bounds(on), "bitsmoe_debug_bounds")


def bitsmoe_debug_shift_expert_records(layer, e: int, delta: int) -> None:
    """Testing hook: shift the code offsets of expert e's gate/up staging records by delta bytes."""
    _check(_lib().bitsmoe_debug_shift_expert_records(layer.handle, e, delta), "bitsmoe_debug_shift_expert_records")


def bitsmoe_debug_wait_limit(skip_arrival: int, spin_clocks: int) -> None:
    """Testing hook: bound the fused kernels' waits to spin_clocks SM clocks (0: default) and let
    block 0 skip its first grid-barrier arrival (skip_arrival = 1)."""
    _check(_lib().bitsmoe_debug_wait_limit(skip_arrival, spin_clocks), "bitsmoe_debug_wait_limit")
