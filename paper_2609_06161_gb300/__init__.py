"""GB300 (sm_103a) AF1 binary-factorized linear layer.

Thin ctypes binding over libaf1.so, whose C ABI is include/af1.h. The binding
only marshals arguments: PyTorch supplies device memory and the current
stream, and every step of the forward pass runs in the library's CUDA
kernels. There is no CPU or PyTorch fallback: if libaf1.so is missing this
package fails to import.

The layer (AF1, Sec. 3.1, Eq. final_reconstruction) is
    W_hat = Diag(a) U Diag(s) V^T Diag(b),     y = x W_hat^T
with U (m x r) and V (n x r) sign matrices, FP16 scales a (m), s (r), b (n).
"""
from __future__ import annotations

import ctypes
import os

import torch

__all__ = [
    "AF1Error", "Layer", "Step", "rank_for_budget", "workspace_status", "static_status", "last_error", "version",
    "lib_path", "words_per_row", "set_wait_cycles", "get_wait_cycles", "AF1_F16", "AF1_F32",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
lib_path = os.path.join(_HERE, "libaf1.so")

if not os.path.exists(lib_path):
    raise ImportError(
        f"{lib_path} is missing: build it with `python paper_2609_06161_gb300/build.py` "
        "(or __graft_entry__.build()); there is no fallback implementation")

_lib = ctypes.CDLL(lib_path)

AF1_OK = 0
AF1_F16 = 0
AF1_F32 = 1
AF1_FLAG_ANY_RANK = 1
AF1_FLAG_TC_DECODE = 2
AF1_FLAG_BF16_SCALES = 4
AF1_FLAG_STREAM_DECODE = 8
AF1_FLAG_MMA_DECODE = 16
AF1_FLAG_LUT_DECODE = 32


def _flags(any_rank: bool, tc_decode: bool, scales=(), stream_decode: bool = False, mma_decode: bool = False,
           lut_decode: bool = False) -> int:
    """Layer flags; BF16 scale tensors select AF1_FLAG_BF16_SCALES."""
    dts = {t.dtype for t in scales}
    if len(dts) > 1 or not dts <= {torch.float16, torch.bfloat16}:
        raise ValueError("a, s and b must all be float16 or all bfloat16")
    bf16 = dts == {torch.bfloat16}
    return ((AF1_FLAG_ANY_RANK if any_rank else 0) | (AF1_FLAG_TC_DECODE if tc_decode else 0)
            | (AF1_FLAG_BF16_SCALES if bf16 else 0) | (AF1_FLAG_STREAM_DECODE if stream_decode else 0)
            | (AF1_FLAG_MMA_DECODE if mma_decode else 0) | (AF1_FLAG_LUT_DECODE if lut_decode else 0))
_ERR_NAMES = {
    -1: "AF1_ERR_INVALID_ARG", -2: "AF1_ERR_BAD_POINTER", -3: "AF1_ERR_MISALIGNED",
    -4: "AF1_ERR_OVER_BUDGET", -5: "AF1_ERR_INVALID_SIGN", -6: "AF1_ERR_CUDA",
    -7: "AF1_ERR_TIMEOUT", -8: "AF1_ERR_WORKSPACE",
}


class _Desc(ctypes.Structure):
    _fields_ = [("m", ctypes.c_int64), ("n", ctypes.c_int64), ("r", ctypes.c_int64),
                ("flags", ctypes.c_int32), ("reserved", ctypes.c_int32)]


_vp = ctypes.c_void_p
_i64 = ctypes.c_int64
_lib.af1_rank_for_budget.argtypes = [_i64, _i64, _i64, _i64, ctypes.POINTER(_i64)]
_lib.af1_rank_for_budget.restype = ctypes.c_int
_lib.af1_storage_bits.argtypes = [_i64, _i64, _i64, ctypes.POINTER(_i64)]
_lib.af1_storage_bits.restype = ctypes.c_int
_lib.af1_pack_layer.argtypes = [ctypes.POINTER(_Desc), _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                ctypes.POINTER(_vp)]
_lib.af1_pack_layer.restype = ctypes.c_int
_lib.af1_load_packed_layer.argtypes = [ctypes.POINTER(_Desc), _vp, _vp, _vp, _vp, _vp, _vp,
                                       ctypes.POINTER(_vp)]
_lib.af1_load_packed_layer.restype = ctypes.c_int
_lib.af1_layer_get_desc.argtypes = [_vp, ctypes.POINTER(_Desc)]
_lib.af1_layer_get_desc.restype = ctypes.c_int
_lib.af1_layer_device_bytes.argtypes = [_vp, ctypes.POINTER(_i64), ctypes.POINTER(_i64)]
_lib.af1_layer_device_bytes.restype = ctypes.c_int
_lib.af1_workspace_bytes.argtypes = [_vp, _i64]
_lib.af1_workspace_bytes.restype = _i64
_lib.af1_linear_forward.argtypes = [_vp, _vp, _i64, _i64, _vp, _i64, ctypes.c_int, _vp, _i64, _vp]
_lib.af1_linear_forward.restype = ctypes.c_int
_lib.af1_workspace_bytes_swiglu.argtypes = [_vp, _i64]
_lib.af1_workspace_bytes_swiglu.restype = _i64
_lib.af1_linear_forward_swiglu.argtypes = [_vp, _vp, _vp, _i64, _i64, _vp, _i64, ctypes.c_int, _vp, _i64, _vp]
_lib.af1_linear_forward_swiglu.restype = ctypes.c_int
_lib.af1_workspace_bytes_multi.argtypes = [ctypes.POINTER(_vp), ctypes.c_int, _i64]
_lib.af1_workspace_bytes_multi.restype = _i64
_lib.af1_linear_forward_multi.argtypes = [ctypes.POINTER(_vp), ctypes.c_int, _vp, _i64, _i64, ctypes.POINTER(_vp),
                                          ctypes.POINTER(_i64), ctypes.c_int, _vp, _i64, _vp]
_lib.af1_linear_forward_multi.restype = ctypes.c_int
_lib.af1_export_layer.argtypes = [_vp, _vp, _vp, _vp, _vp, _vp, _vp]
_lib.af1_export_layer.restype = ctypes.c_int
_lib.af1_save_layer.argtypes = [_vp, ctypes.c_char_p]
_lib.af1_save_layer.restype = ctypes.c_int
_lib.af1_load_layer.argtypes = [ctypes.c_char_p, _vp, ctypes.POINTER(_vp)]
_lib.af1_load_layer.restype = ctypes.c_int
_dp = ctypes.POINTER(ctypes.c_double)
_lib.af1_hisa_layer_budgets.argtypes = [_dp, _i64, ctypes.c_double, ctypes.c_double, _dp]
_lib.af1_hisa_layer_budgets.restype = ctypes.c_int
_lib.af1_hisa_module_budgets.argtypes = [_dp, _dp, ctypes.POINTER(_i64), _i64, ctypes.c_double, ctypes.c_double,
                                         ctypes.c_double, _dp]
_lib.af1_hisa_module_budgets.restype = ctypes.c_int
_lib.af1_budget_to_rank.argtypes = [ctypes.c_double, _i64, _i64, ctypes.POINTER(_i64)]
_lib.af1_budget_to_rank.restype = ctypes.c_int


class _NabfParams(ctypes.Structure):
    _fields_ = [("iters", ctypes.c_int32), ("power_iters", ctypes.c_int32), ("rho", ctypes.c_double),
                ("eta", ctypes.c_double), ("eps", ctypes.c_double), ("seed", ctypes.c_uint64),
                ("compensate", ctypes.c_int32), ("reserved", ctypes.c_int32)]


_lib.af1_nabf_factorize.argtypes = [_vp, _i64, _i64, _i64, _vp, _vp, ctypes.POINTER(_NabfParams), _vp, _vp, _vp,
                                    _vp, _vp, _dp, _vp]
_lib.af1_nabf_factorize.restype = ctypes.c_int
_lib.af1_workspace_status.argtypes = [_vp, _vp]
_lib.af1_workspace_status.restype = ctypes.c_int
_lib.af1_static_status.argtypes = [_vp]
_lib.af1_static_status.restype = ctypes.c_int
_lib.af1_set_wait_cycles.argtypes = [_i64]
_lib.af1_set_wait_cycles.restype = ctypes.c_int
_lib.af1_get_wait_cycles.argtypes = []
_lib.af1_get_wait_cycles.restype = _i64
_lib.af1_mma_plan_dry.argtypes = [ctypes.c_int, _i64, _i64, _i64, ctypes.c_int, ctypes.c_int,
                                  ctypes.POINTER(ctypes.c_int32)]
_lib.af1_mma_plan_dry.restype = ctypes.c_int
_lib.af1_set_stream_layout.argtypes = [ctypes.c_int]
_lib.af1_set_stream_layout.restype = ctypes.c_int
_lib.af1_get_stream_layout.argtypes = []
_lib.af1_get_stream_layout.restype = ctypes.c_int


class _StepLinear(ctypes.Structure):
    _fields_ = [("layer", _vp), ("x", _vp), ("x2", _vp), ("ldx", _i64), ("y", _vp), ("ldy", _i64),
                ("level", ctypes.c_int32), ("reserved", ctypes.c_int32)]


_lib.af1_step_create.argtypes = [ctypes.POINTER(_StepLinear), ctypes.c_int, _i64, ctypes.c_int, ctypes.c_int32,
                                 ctypes.POINTER(_vp)]
_lib.af1_step_create.restype = ctypes.c_int
_lib.af1_step_workspace_bytes.argtypes = [_vp]
_lib.af1_step_workspace_bytes.restype = _i64
_lib.af1_step_info.argtypes = [_vp, ctypes.POINTER(_i64), ctypes.POINTER(_i64), ctypes.POINTER(_i64),
                               ctypes.POINTER(ctypes.c_double)]
_lib.af1_step_info.restype = ctypes.c_int
_lib.af1_step_run.argtypes = [_vp, _vp, _i64, _vp]
_lib.af1_step_run.restype = ctypes.c_int
_lib.af1_step_open_gate.argtypes = [_vp, _vp]
_lib.af1_step_open_gate.restype = ctypes.c_int
_lib.af1_step_destroy.argtypes = [_vp]
_lib.af1_step_destroy.restype = None
_lib.af1_free.argtypes = [_vp]
_lib.af1_free.restype = None
_lib.af1_last_error.argtypes = []
_lib.af1_last_error.restype = ctypes.c_char_p
_lib.af1_version.argtypes = []
_lib.af1_version.restype = ctypes.c_char_p


class AF1Error(RuntimeError):
    def __init__(self, code: int, message: str):
        self.code = code
        self.name = _ERR_NAMES.get(code, str(code))
        super().__init__(f"{self.name}: {message}")


def last_error() -> str:
    return _lib.af1_last_error().decode()


def version() -> str:
    return _lib.af1_version().decode()


def _check(rc: int):
    if rc != AF1_OK:
        raise AF1Error(rc, last_error())


def words_per_row(cols: int) -> int:
    """uint32 words per packed row of `cols` signs (rows padded to 16 bytes)."""
    return 4 * ((cols + 127) // 128)


def rank_for_budget(m: int, n: int, num: int = 1, den: int = 1) -> int:
    """Largest r whose exact AF1 storage fits num/den bits per weight."""
    r = _i64(0)
    _check(_lib.af1_rank_for_budget(m, n, num, den, ctypes.byref(r)))
    return r.value


def storage_bits(m: int, n: int, r: int) -> int:
    """Bits one layer stores: r(m+n) signs plus m + r + n FP16 scales."""
    b = _i64(0)
    _check(_lib.af1_storage_bits(m, n, r, ctypes.byref(b)))
    return b.value


def _stream_handle(stream) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return int(s.cuda_stream)


def _ptr(t) -> int:
    return 0 if t is None else int(t.data_ptr())


def workspace_status(workspace: torch.Tensor, stream=None) -> None:
    """Synchronize and raise AF1Error(AF1_ERR_TIMEOUT) if a bounded device wait gave up."""
    _check(_lib.af1_workspace_status(_ptr(workspace), _stream_handle(stream)))


def static_status(stream=None) -> None:
    """af1_static_status: raise AF1Error(AF1_ERR_TIMEOUT) if a wait of a
    call of af1_linear_forward_static gave up (the array is then reset)."""
    _check(_lib.af1_static_status(_stream_handle(stream)))


def set_wait_cycles(cycles: int) -> None:
    """Budget (clock64 cycles) of every bounded device wait of later launches."""
    _check(_lib.af1_set_wait_cycles(int(cycles)))


def get_wait_cycles() -> int:
    return int(_lib.af1_get_wait_cycles())


def mma_plan_dry(phase: int, R: int, C: int, tokens: int, num_sms: int = 152, max_smem: int = 232448) -> dict:
    """The 16-bit-operand decode kernel's launch plan for one phase (an R x C
    sign matrix times `tokens` vectors), computed on the host
    (af1_mma_plan_dry); no GPU needed."""
    out = (ctypes.c_int32 * 10)()
    _check(_lib.af1_mma_plan_dry(int(phase), int(R), int(C), int(tokens), int(num_sms), int(max_smem), out))
    keys = ("rows", "accumulators", "ring", "tmem_cols", "ks", "cpc", "smem", "grid_x", "grid_y", "ok")
    return dict(zip(keys, list(out)))


AF1_ONE_STREAM = 0
AF1_MANY_STREAMS = 1


def set_stream_layout(layout: int) -> None:
    """AF1_ONE_STREAM (default: calls one after another on one stream) or
    AF1_MANY_STREAMS (several streams run layers at once); the lookup-table
    decode kernels adapt their launch order and CTA count to it
    (af1_set_stream_layout)."""
    _check(_lib.af1_set_stream_layout(int(layout)))


def get_stream_layout() -> int:
    return int(_lib.af1_get_stream_layout())


class Layer:
    """An AF1 layer resident on the current CUDA device."""

    def __init__(self, handle: int, m: int, n: int, r: int):
        self._h = handle
        self.m, self.n, self.r = m, n, r

    # -- construction --------------------------------------------------------
    @classmethod
    def from_signs(cls, U: torch.Tensor, V: torch.Tensor, a: torch.Tensor, s: torch.Tensor,
                   b: torch.Tensor, any_rank: bool = False, return_words: bool = False, stream=None,
                   tc_decode: bool = False, stream_decode: bool = False, mma_decode: bool = False,
                   lut_decode: bool = False):
        """U: int8 (m, r), V: int8 (n, r) of +-1; a, s, b: float16 vectors. All on
        the current CUDA device. With return_words, also returns the canonical
        packed words (Uw: (m, W(r)), Vw: (r, W(n)) as int32 tensors). tc_decode
        selects the e4m3 tensor-core decode kernel (AF1_FLAG_TC_DECODE),
        mma_decode the 16-bit-operand tensor-core decode kernel for every pass
        (AF1_FLAG_MMA_DECODE), lut_decode the lookup-table kernels for every
        pass (AF1_FLAG_LUT_DECODE), stream_decode the streaming CUDA-core kernel
        for 1- and 2-token passes (AF1_FLAG_STREAM_DECODE)."""
        m, r = U.shape
        n = V.shape[0]
        if V.shape[1] != r:
            raise ValueError("U and V must have the same rank")
        U, V = U.contiguous(), V.contiguous()
        a, s, b = a.contiguous(), s.contiguous(), b.contiguous()
        Uw = Vw = None
        if return_words:
            Uw = torch.empty((m, words_per_row(r)), dtype=torch.int32, device=U.device)
            Vw = torch.empty((r, words_per_row(n)), dtype=torch.int32, device=U.device)
        d = _Desc(m, n, r, _flags(any_rank, tc_decode, (a, s, b), stream_decode, mma_decode, lut_decode), 0)
        h = _vp()
        _check(_lib.af1_pack_layer(ctypes.byref(d), _ptr(U), _ptr(V), _ptr(a), _ptr(s), _ptr(b),
                                   _ptr(Uw), _ptr(Vw), _stream_handle(stream), ctypes.byref(h)))
        layer = cls(h.value, m, n, r)
        return (layer, Uw, Vw) if return_words else layer

    @classmethod
    def from_words(cls, Uw: torch.Tensor, Vw: torch.Tensor, a: torch.Tensor, s: torch.Tensor,
                   b: torch.Tensor, m: int, n: int, r: int, any_rank: bool = False, stream=None,
                   tc_decode: bool = False, stream_decode: bool = False, mma_decode: bool = False,
                   lut_decode: bool = False):
        """Uw: (m, W(r)), Vw: (r, W(n)) canonical packed words (int32/uint32)."""
        Uw, Vw = Uw.contiguous(), Vw.contiguous()
        a, s, b = a.contiguous(), s.contiguous(), b.contiguous()
        d = _Desc(m, n, r, _flags(any_rank, tc_decode, (a, s, b), stream_decode, mma_decode, lut_decode), 0)
        h = _vp()
        _check(_lib.af1_load_packed_layer(ctypes.byref(d), _ptr(Uw), _ptr(Vw), _ptr(a), _ptr(s), _ptr(b),
                                          _stream_handle(stream), ctypes.byref(h)))
        return cls(h.value, m, n, r)

    @classmethod
    def load(cls, path: str, stream=None):
        """A layer from a file written by save() (af1_load_layer)."""
        h = _vp()
        _check(_lib.af1_load_layer(str(path).encode(), _stream_handle(stream), ctypes.byref(h)))
        d = _Desc()
        _check(_lib.af1_layer_get_desc(h, ctypes.byref(d)))
        return cls(h.value, d.m, d.n, d.r)

    def save(self, path: str) -> None:
        """Write the layer to a file (af1_save_layer; format in include/af1.h)."""
        _check(_lib.af1_save_layer(self._h, str(path).encode()))

    def export(self, stream=None):
        """(Uw, Vw, a, s, b): canonical packed words (int32, (m, W(r)) and
        (r, W(n))) and FP16 scales, on the layer's device (af1_export_layer)."""
        dev = torch.device("cuda", torch.cuda.current_device())
        Uw = torch.empty((self.m, words_per_row(self.r)), dtype=torch.int32, device=dev)
        Vw = torch.empty((self.r, words_per_row(self.n)), dtype=torch.int32, device=dev)
        a = torch.empty(self.m, dtype=torch.float16, device=dev)
        s = torch.empty(self.r, dtype=torch.float16, device=dev)
        b = torch.empty(self.n, dtype=torch.float16, device=dev)
        _check(_lib.af1_export_layer(self._h, _ptr(Uw), _ptr(Vw), _ptr(a), _ptr(s), _ptr(b), _stream_handle(stream)))
        return Uw, Vw, a, s, b

    # -- queries ---------------------------------------------------------------
    def workspace_bytes(self, tokens: int = 1) -> int:
        v = _lib.af1_workspace_bytes(self._h, tokens)
        if v < 0:
            raise AF1Error(int(v), last_error())
        return int(v)

    def make_workspace(self, tokens: int = 16, device=None) -> torch.Tensor:
        """A zero-filled workspace tensor usable for any number of tokens."""
        return torch.zeros(self.workspace_bytes(tokens), dtype=torch.uint8,
                           device=device or torch.device("cuda", torch.cuda.current_device()))

    def device_bytes(self):
        sb, cb = _i64(0), _i64(0)
        _check(_lib.af1_layer_device_bytes(self._h, ctypes.byref(sb), ctypes.byref(cb)))
        return sb.value, cb.value

    # -- compute -----------------------------------------------------------------
    def forward_into(self, x: torch.Tensor, y: torch.Tensor, workspace: torch.Tensor, stream=None) -> None:
        """y[:tokens, :m] = x[:tokens, :n] W_hat^T; x float16 (tokens, ldx),
        y float16 or float32 (tokens, ldy), both 2-D with unit column stride."""
        if x.dim() != 2 or y.dim() != 2 or x.stride(1) != 1 or y.stride(1) != 1:
            raise ValueError("x and y must be 2-D with contiguous rows")
        if x.dtype != torch.float16:
            raise ValueError("x must be float16")
        if y.dtype == torch.float16:
            yd = AF1_F16
        elif y.dtype == torch.float32:
            yd = AF1_F32
        else:
            raise ValueError("y must be float16 or float32")
        tokens = x.shape[0]
        if y.shape[0] < tokens:
            raise ValueError("y has fewer rows than x")
        ldx = x.stride(0) if tokens > 1 else max(x.stride(0), self.n + (-self.n) % 8)
        ldy = y.stride(0) if tokens > 1 else max(y.stride(0), self.m + (-self.m) % (8 if yd == AF1_F16 else 4))
        _check(_lib.af1_linear_forward(self._h, _ptr(x), ldx, tokens, _ptr(y), ldy, yd, _ptr(workspace),
                                       workspace.numel() * workspace.element_size(), _stream_handle(stream)))

    def forward(self, x: torch.Tensor, out_dtype=torch.float16, workspace: torch.Tensor | None = None,
                stream=None) -> torch.Tensor:
        if x.dim() == 1:
            x = x.unsqueeze(0)
        tokens = x.shape[0]
        if x.stride(1) != 1 or x.stride(0) % 8 != 0 or x.data_ptr() % 16 != 0:
            pad = (-self.n) % 8
            xp = torch.zeros((tokens, self.n + pad), dtype=torch.float16, device=x.device)
            xp[:, :self.n] = x
            x = xp
        align = 8 if out_dtype == torch.float16 else 4
        ldy = self.m + (-self.m) % align
        y = torch.empty((tokens, ldy), dtype=out_dtype, device=x.device)
        ws = workspace if workspace is not None else self.make_workspace(tokens, x.device)
        self.forward_into(x, y, ws, stream)
        return y[:, :self.m]

    def workspace_bytes_swiglu(self, tokens: int = 1) -> int:
        v = _lib.af1_workspace_bytes_swiglu(self._h, tokens)
        if v < 0:
            raise AF1Error(int(v), last_error())
        return int(v)

    def forward_swiglu_into(self, g: torch.Tensor, u: torch.Tensor, y: torch.Tensor, workspace: torch.Tensor,
                            stream=None) -> None:
        """y[:tokens, :m] = h W_hat^T with h = FP16(SiLU(g) * u)
        (af1_linear_forward_swiglu); g and u float16 (tokens, ldx) with the
        same strides, y float16 or float32 (tokens, ldy)."""
        for t in (g, u, y):
            if t.dim() != 2 or t.stride(1) != 1:
                raise ValueError("g, u and y must be 2-D with contiguous rows")
        if g.dtype != torch.float16 or u.dtype != torch.float16:
            raise ValueError("g and u must be float16")
        if g.shape != u.shape or g.stride() != u.stride():
            raise ValueError("g and u must have the same shape and strides")
        if y.dtype == torch.float16:
            yd = AF1_F16
        elif y.dtype == torch.float32:
            yd = AF1_F32
        else:
            raise ValueError("y must be float16 or float32")
        tokens = g.shape[0]
        if y.shape[0] < tokens:
            raise ValueError("y has fewer rows than g")
        ldx = g.stride(0) if tokens > 1 else max(g.stride(0), self.n + (-self.n) % 8)
        ldy = y.stride(0) if tokens > 1 else max(y.stride(0), self.m + (-self.m) % (8 if yd == AF1_F16 else 4))
        _check(_lib.af1_linear_forward_swiglu(self._h, _ptr(g), _ptr(u), ldx, tokens, _ptr(y), ldy, yd,
                                              _ptr(workspace), workspace.numel() * workspace.element_size(),
                                              _stream_handle(stream)))

    def forward_swiglu(self, g: torch.Tensor, u: torch.Tensor, out_dtype=torch.float16,
                       workspace: torch.Tensor | None = None, stream=None) -> torch.Tensor:
        if g.dim() == 1:
            g, u = g.unsqueeze(0), u.unsqueeze(0)
        tokens = g.shape[0]
        pad = (-self.n) % 8
        gp = torch.zeros((tokens, self.n + pad), dtype=torch.float16, device=g.device)
        up = torch.zeros_like(gp)
        gp[:, :self.n] = g
        up[:, :self.n] = u
        align = 8 if out_dtype == torch.float16 else 4
        y = torch.empty((tokens, self.m + (-self.m) % align), dtype=out_dtype, device=g.device)
        ws = workspace if workspace is not None else torch.zeros(self.workspace_bytes_swiglu(tokens),
                                                                 dtype=torch.uint8, device=g.device)
        self.forward_swiglu_into(gp, up, y, ws, stream)
        return y[:, :self.m]

    def free(self) -> None:
        if getattr(self, "_h", None):
            _lib.af1_free(self._h)
            self._h = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


# -- several layers sharing their input ------------------------------------------

def workspace_bytes_multi(layers, tokens: int = 1) -> int:
    """Workspace bytes of forward_multi over `layers` (1..4 Layer objects)."""
    arr = (_vp * len(layers))(*[L._h for L in layers])
    v = _lib.af1_workspace_bytes_multi(arr, len(layers), tokens)
    if v < 0:
        raise AF1Error(int(v), last_error())
    return int(v)


def forward_multi(layers, x: torch.Tensor, ys, workspace: torch.Tensor, stream=None) -> None:
    """ys[i][:tokens, :m_i] = x[:tokens, :n] W_hat_i^T for layers with the same
    n (af1_linear_forward_multi); x float16 (tokens, ldx), every ys[i] float16
    or every one float32, all 2-D with unit column stride."""
    if x.dim() != 2 or x.stride(1) != 1 or x.dtype != torch.float16:
        raise ValueError("x must be 2-D float16 with contiguous rows")
    if len(ys) != len(layers):
        raise ValueError("one output per layer")
    yd = AF1_F16 if ys[0].dtype == torch.float16 else AF1_F32
    tokens = x.shape[0]
    n = layers[0].n
    ldx = x.stride(0) if tokens > 1 else max(x.stride(0), n + (-n) % 8)
    ldys = []
    for L, y in zip(layers, ys):
        if y.dim() != 2 or y.stride(1) != 1 or y.shape[0] < tokens:
            raise ValueError("every y must be 2-D with contiguous rows and at least `tokens` rows")
        if (y.dtype == torch.float16) != (yd == AF1_F16) or y.dtype not in (torch.float16, torch.float32):
            raise ValueError("outputs must all be float16 or all float32")
        align = 8 if yd == AF1_F16 else 4
        ldys.append(y.stride(0) if tokens > 1 else max(y.stride(0), L.m + (-L.m) % align))
    hs = (_vp * len(layers))(*[L._h for L in layers])
    yp = (_vp * len(ys))(*[_ptr(y) for y in ys])
    ld = (_i64 * len(ys))(*ldys)
    _check(_lib.af1_linear_forward_multi(hs, len(layers), _ptr(x), ldx, tokens, yp, ld, yd, _ptr(workspace),
                                         workspace.numel() * workspace.element_size(), _stream_handle(stream)))


# -- HiSA budget arithmetic (host) --------------------------------------------------

def _dbl(v):
    a = (ctypes.c_double * len(v))(*[float(x) for x in v])
    return a


def hisa_layer_budgets(phi, B_total: float, tau: float = 1.0):
    """Layer budgets from layer Shapley scores (af1_hisa_layer_budgets)."""
    out = (ctypes.c_double * len(phi))()
    _check(_lib.af1_hisa_layer_budgets(_dbl(phi), len(phi), B_total, tau, out))
    return list(out)


def hisa_module_budgets(phi_dir, phi_mag, params, B_l: float, alpha: float = 0.2, eps: float = 1e-8):
    """Module budgets (bits per weight) within one layer (af1_hisa_module_budgets)."""
    n = len(params)
    if len(phi_dir) != n or len(phi_mag) != n:
        raise ValueError("one score pair per module")
    out = (ctypes.c_double * n)()
    p = (_i64 * n)(*[int(x) for x in params])
    _check(_lib.af1_hisa_module_budgets(_dbl(phi_dir), _dbl(phi_mag), p, n, B_l, alpha, eps, out))
    return list(out)


def budget_to_rank(b: float, m: int, n: int) -> int:
    """r = Round(b m n / (m + n)), clipped to [1, 32768] (af1_budget_to_rank)."""
    r = _i64()
    _check(_lib.af1_budget_to_rank(b, m, n, ctypes.byref(r)))
    return r.value


# -- NABF: factorize a weight matrix into an AF1 layer -----------------------------

def nabf_factorize(W: torch.Tensor, r: int, iters: int = 10, rho: float = 1.0, eta: float = 0.01,
                   eps: float = 1e-8, power_iters: int = 20, seed: int = 0, in_scale=None, out_scale=None,
                   compensate: bool = True, stream=None) -> dict:
    """Algorithm NABF on W (float32 CUDA tensor, m x n) at rank r
    (af1_nabf_factorize). Returns U (int8 m x r), V (int8 n x r), a, s, b
    (float32, the surrogate scaling undone), the relative objective per
    iteration and the null-space sizes kept per iteration (left, right)."""
    W = W.contiguous().float()
    m, n = W.shape
    dev = W.device
    U = torch.empty((m, r), dtype=torch.int8, device=dev)
    V = torch.empty((n, r), dtype=torch.int8, device=dev)
    a = torch.empty(m, dtype=torch.float32, device=dev)
    s_ = torch.empty(r, dtype=torch.float32, device=dev)
    b = torch.empty(n, dtype=torch.float32, device=dev)
    i_s = None if in_scale is None else in_scale.contiguous().float()
    o_s = None if out_scale is None else out_scale.contiguous().float()
    hist = (ctypes.c_double * (3 * (iters + 1)))()
    p = _NabfParams(iters, power_iters, rho, eta, eps, seed & ((1 << 64) - 1), 1 if compensate else 0, 0)
    _check(_lib.af1_nabf_factorize(_ptr(W), m, n, r, _ptr(i_s), _ptr(o_s), ctypes.byref(p), _ptr(U), _ptr(V),
                                   _ptr(a), _ptr(s_), _ptr(b), hist, _stream_handle(stream)))
    h = list(hist)
    k = iters + 1
    return {"U": U, "V": V, "a": a, "s": s_, "b": b, "objective": h[:k], "q_left": [int(v) for v in h[k:2 * k]],
            "q_right": [int(v) for v in h[2 * k:]]}


# -- a decode step as one launch -------------------------------------------------------

AF1_STEP_WAIT_GATE = 1


def _row_stride(t: torch.Tensor, cols: int, align: int) -> int:
    if t.dim() != 2 or t.stride(1) != 1:
        raise ValueError("step tensors must be 2-D with contiguous rows")
    return t.stride(0) if t.shape[0] > 1 else max(t.stride(0), cols + (-cols) % align)


class Step:
    """af1_step_*: many linears in dependent levels as one persistent launch.

    linears: sequence of (layer, x, y, level) or (layer, x, y, level, x2)
    tuples; x (and x2, the `up` output of a SwiGLU input) float16
    (tokens, ldx), y float16 or float32 (tokens, ldy), all on the current
    device. The tensors are kept alive by this object; every run reads the
    x buffers and writes the y buffers given here."""

    def __init__(self, linears, gate: bool = False):
        items = []
        keep = []
        tokens = None
        ydt = None
        for item in linears:
            layer, x, y, level = item[:4]
            x2 = item[4] if len(item) > 4 else None
            if x.dtype != torch.float16 or (x2 is not None and x2.dtype != torch.float16):
                raise ValueError("x and x2 must be float16")
            if y.dtype not in (torch.float16, torch.float32):
                raise ValueError("y must be float16 or float32")
            ydt = ydt or y.dtype
            if y.dtype != ydt:
                raise ValueError("all outputs must have one dtype")
            tokens = tokens or x.shape[0]
            if x.shape[0] != tokens or y.shape[0] < tokens:
                raise ValueError("all inputs must have the same number of rows")
            yd = AF1_F16 if ydt == torch.float16 else AF1_F32
            ldx = _row_stride(x, layer.n, 8)
            if x2 is not None and (x2.shape != x.shape or x2.stride() != x.stride()):
                raise ValueError("x2 must have the shape and strides of x")
            ldy = _row_stride(y, layer.m, 8 if yd == AF1_F16 else 4)
            items.append(_StepLinear(layer._h, _ptr(x), _ptr(x2), ldx, _ptr(y), ldy, int(level), 0))
            keep += [layer, x, y, x2]
        arr = (_StepLinear * len(items))(*items)
        h = _vp()
        yd = AF1_F16 if ydt == torch.float16 else AF1_F32
        _check(_lib.af1_step_create(arr, len(items), tokens, yd, AF1_STEP_WAIT_GATE if gate else 0,
                                    ctypes.byref(h)))
        self._h = h.value
        self._keep = keep
        self.tokens = tokens

    def workspace_bytes(self) -> int:
        v = _lib.af1_step_workspace_bytes(self._h)
        if v < 0:
            raise AF1Error(int(v), last_error())
        return int(v)

    def make_workspace(self, device=None) -> torch.Tensor:
        return torch.zeros(self.workspace_bytes(), dtype=torch.uint8,
                           device=device or torch.device("cuda", torch.cuda.current_device()))

    def info(self) -> dict:
        c, t, lv, us = _i64(), _i64(), _i64(), ctypes.c_double()
        _check(_lib.af1_step_info(self._h, ctypes.byref(c), ctypes.byref(t), ctypes.byref(lv), ctypes.byref(us)))
        return {"ctas": c.value, "tasks": t.value, "levels": lv.value, "model_us": us.value}

    def run(self, workspace: torch.Tensor, stream=None) -> None:
        _check(_lib.af1_step_run(self._h, _ptr(workspace), workspace.numel() * workspace.element_size(),
                                 _stream_handle(stream)))

    @staticmethod
    def open_gate(workspace: torch.Tensor, stream=None) -> None:
        _check(_lib.af1_step_open_gate(_ptr(workspace), _stream_handle(stream)))

    def destroy(self) -> None:
        if getattr(self, "_h", None):
            _lib.af1_step_destroy(self._h)
            self._h = None
            self._keep = []

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass
