"""Python binding of the libpatconv C ABI (argument marshalling only).

``pp_pack`` / ``pp_conv`` / ``pp_maxpool2x2`` mirror the C entry points of include/patconv.h;
``Layer`` owns a packed-layer handle and the device buffer its image is bound to.  PyTorch is
used for device memory and streams only: every step of the convolution runs in the library's
CUDA kernels, and a non-CUDA tensor is rejected rather than computed elsewhere.
"""
from __future__ import annotations

import ctypes
from typing import Optional, Sequence

import numpy as np
import torch

from . import _lib

PP_F32, PP_F16 = 0, 1
SECTIONS = {"header": 0, "pid": 1, "perm": 2, "desc": 3, "kofs": 4, "vals": 5, "dense": 6,
            "image": 7}
SECTION_DTYPES = {"header": np.uint32, "pid": np.int8, "perm": np.uint32, "desc": np.uint64,
                  "kofs": np.uint32, "vals": np.float32, "dense": np.float32, "image": np.uint8}
QUERY = {"beta": 0, "cout": 1, "cin_g": 2, "groups": 3, "stride": 4, "n_groups": 5,
         "n_patterns": 6, "image_bytes": 7, "fast_path": 8}
_DT = {torch.float32: PP_F32, torch.float16: PP_F16}


def default_patterns() -> list:
    """The 8-pattern library the kernels are compiled for (9-bit raster masks)."""
    buf = (ctypes.c_uint16 * 8)()
    n = _lib.load().pp_default_patterns(buf, 8)
    return [int(buf[i]) for i in range(n)]


def _stream_ptr(stream, device) -> ctypes.c_void_p:
    s = stream if stream is not None else torch.cuda.current_stream(device)
    return ctypes.c_void_p(int(s.cuda_stream))


class Layer:
    """A packed pattern-pruned 3x3 layer (handle of pp_pack)."""

    def __init__(self, handle: ctypes.c_void_p):
        self._h = handle
        self._dev_buf: Optional[torch.Tensor] = None

    # ---- host side
    def query(self, key: str) -> int:
        v = ctypes.c_int64()
        _lib.check("pp_query", _lib.load().pp_query(self._h, QUERY[key], ctypes.byref(v)))
        return int(v.value)

    def section_bytes(self, name: str) -> int:
        v = ctypes.c_int64()
        _lib.check("pp_query", _lib.load().pp_query(self._h, 16 + SECTIONS[name], ctypes.byref(v)))
        return int(v.value)

    def export(self, name: str) -> np.ndarray:
        n = self.section_bytes(name)
        out = np.zeros(n, dtype=np.uint8)
        _lib.check("pp_export", _lib.load().pp_export(self._h, SECTIONS[name],
                                                      out.ctypes.data_as(ctypes.c_void_p), n))
        return out.view(SECTION_DTYPES[name])

    @property
    def beta(self) -> int:
        return self.query("beta")

    @property
    def cout(self) -> int:
        return self.query("cout")

    @property
    def cin_g(self) -> int:
        return self.query("cin_g")

    @property
    def stride(self) -> int:
        return self.query("stride")

    @property
    def depthwise(self) -> bool:
        return self.query("groups") != 1

    # ---- device side
    def bind(self, device=None, stream=None) -> "Layer":
        """Copy the device image into a fresh torch buffer on ``device`` (async on ``stream``)."""
        device = torch.device(device if device is not None else "cuda")
        if device.type != "cuda":
            raise ValueError("the packed image must live in CUDA device memory")
        n = self.query("image_bytes")
        buf = torch.empty(n, dtype=torch.uint8, device=device)
        _lib.check("pp_bind_device", _lib.load().pp_bind_device(
            self._h, ctypes.c_void_p(buf.data_ptr()), n, _stream_ptr(stream, device)))
        self._dev_buf = buf
        return self

    def out_shape(self, x_shape) -> tuple:
        N, _, H, W = x_shape
        s = self.stride
        return (N, self.cout, (H - 1) // s + 1, (W - 1) // s + 1)

    PLAN_KEYS = ("path", "splits", "workspace_bytes", "units", "tile_by", "tile_bx", "tile_nb",
                 "channels_per_stage", "filter_groups", "spatial_warps", "smem_bytes",
                 "chunks_per_unit", "ctas", "lane_sort", "shift", "streamk", "groups_per_warp")

    def plan(self, x_shape, workspace_bytes: int = 0, pool2x2: bool = False,
             dtype=torch.float32) -> dict:
        """Launch plan pp_conv_ws (or, with pool2x2, pp_conv_pool_ws) would use for an input of
        shape [N, C, H, W] and dtype (pp_conv_plan_dt).  Depthwise layers report ``dw_kernel``:
        1 streamed rows, 2 streamed planes at stride 2, 3 / 4 streamed planes at stride 1 (rows of
        even / odd width), 5 / 6 streamed tiles of 7 / 14 columns at stride 1, 7 streamed tiles at
        stride 2, 0 the row-item kernels (for 16-byte aligned x and y)."""
        N, _, H, W = x_shape
        n = len(self.PLAN_KEYS)
        info = (ctypes.c_int64 * n)()
        _lib.check("pp_conv_plan_dt", _lib.load().pp_conv_plan_dt(
            self._h, _DT[dtype], 1 if pool2x2 else 0, N, H, W, int(workspace_bytes), info, n))
        d = dict(zip(self.PLAN_KEYS, (int(v) for v in info)))
        if d["path"] == 2:   # depthwise: info[1] names the kernel, there is no split
            d = {"path": 2, "splits": 0, "workspace_bytes": 0, "dw_kernel": int(info[1]),
                 "chunks": int(info[3]), "rows_or_planes": int(info[4]), "stages": int(info[5]),
                 "warps": int(info[6]), "smem_bytes": int(info[10]), "ctas": int(info[12])}
        return d

    def workspace_bytes(self, x_shape, pool2x2: bool = False, dtype=torch.float32) -> int:
        """Workspace the call would use for this input shape and dtype (0: none): the input-channel
        split or the balanced schedule, for pp_conv_ws or, with pool2x2, pp_conv_pool_ws."""
        return self.plan(x_shape, (1 << 64) - 1, pool2x2, dtype)["workspace_bytes"]

    def conv(self, x: torch.Tensor, bias: Optional[torch.Tensor] = None, relu: bool = False,
             out: Optional[torch.Tensor] = None, stream=None,
             workspace: Optional[torch.Tensor] = None, pool2x2: bool = False) -> torch.Tensor:
        """y = ReLU?(conv3x3(x, W_hat, stride, pad 1) + bias) via pp_conv_ws; with ``pool2x2``
        the 2x2/2 max-pool of that map, fused into the conv (pp_conv_pool_ws)."""
        if self._dev_buf is None:
            self.bind(x.device)
        if not x.is_cuda or x.dtype not in _DT or not x.is_contiguous() or x.dim() != 4:
            raise ValueError("x must be a contiguous 4-d CUDA float32/float16 tensor (NCHW)")
        cin = self.cout if self.depthwise else self.cin_g
        if x.shape[1] != cin:
            raise ValueError(f"x has {x.shape[1]} channels, layer expects {cin}")
        shape = self.out_shape(tuple(x.shape))
        if pool2x2:
            shape = shape[:2] + (shape[2] // 2, shape[3] // 2)
        if out is None:
            out = torch.empty(shape, dtype=x.dtype, device=x.device)
        if tuple(out.shape) != shape or out.dtype != x.dtype or not out.is_contiguous() or not out.is_cuda:
            raise ValueError(f"out must be a contiguous CUDA tensor of shape {shape} and x's dtype")
        bptr = None
        if bias is not None:
            if not bias.is_cuda or bias.dtype != torch.float32 or bias.numel() != self.cout \
                    or not bias.is_contiguous():
                raise ValueError("bias must be a contiguous CUDA float32 tensor of Cout values")
            bptr = ctypes.c_void_p(bias.data_ptr())
        N, _, H, W = x.shape
        wptr, wbytes = None, 0
        if workspace is not None:
            if not workspace.is_cuda or not workspace.is_contiguous():
                raise ValueError("workspace must be a contiguous CUDA tensor")
            wptr, wbytes = ctypes.c_void_p(workspace.data_ptr()), workspace.numel() * workspace.element_size()
        name = "pp_conv_pool_ws" if pool2x2 else "pp_conv_ws"
        _lib.check(name, getattr(_lib.load(), name)(
            self._h, ctypes.c_void_p(x.data_ptr()), _DT[x.dtype], N, H, W, bptr, int(bool(relu)),
            ctypes.c_void_p(out.data_ptr()), wptr, wbytes, _stream_ptr(stream, x.device)))
        return out

    def __del__(self):
        h, self._h = getattr(self, "_h", None), None
        if h:
            try:
                _lib.load().pp_destroy(h)
            except Exception:
                pass


def design_patterns(weights: Sequence, m: int = 8) -> list:
    """Pattern library of at most m masks from the kernels of ``weights`` (arrays [..., 3, 3]) by
    the §4.2 heuristic (pp_design_patterns): centre + three largest-magnitude taps per kernel,
    the m most frequent of those."""
    W = np.ascontiguousarray(np.concatenate([np.asarray(w, np.float32).reshape(-1, 9) for w in weights]))
    masks = (ctypes.c_uint16 * m)()
    n = ctypes.c_int()
    _lib.check("pp_design_patterns", _lib.load().pp_design_patterns(
        W.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), W.shape[0], m, masks, ctypes.byref(n)))
    return [int(masks[i]) for i in range(n.value)]


def pp_pack(W, pattern_set: Optional[Sequence[int]] = None, keep_ratio: float = 1.0,
            groups: int = 1, stride: int = 1) -> Layer:
    """Pattern projection + connectivity pruning + packing of host weights [Cout, Cin_g, 3, 3]."""
    W = np.ascontiguousarray(np.asarray(W, dtype=np.float32))
    if W.ndim != 4 or W.shape[2:] != (3, 3):
        raise ValueError("W must be [Cout, Cin/groups, 3, 3]")
    masks = list(pattern_set) if pattern_set is not None else default_patterns()
    m = (ctypes.c_uint16 * max(1, len(masks)))(*[int(v) for v in masks])
    cout, cin_g = W.shape[:2]
    cin = cout if groups != 1 else cin_g
    if groups != 1 and cin_g != 1:
        raise ValueError("depthwise weights must be [C, 1, 3, 3]")
    h = ctypes.c_void_p()
    _lib.check("pp_pack", _lib.load().pp_pack(
        W.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), cout, cin, groups, stride, m, len(masks),
        float(keep_ratio), ctypes.byref(h)))
    return Layer(h)


def pp_conv(layer: Layer, x: torch.Tensor, bias: Optional[torch.Tensor], relu: bool,
            y: Optional[torch.Tensor] = None, stream=None,
            workspace: Optional[torch.Tensor] = None) -> torch.Tensor:
    return layer.conv(x, bias, relu, y, stream, workspace)


def workspace_for(layers, x_shapes, device=None, pools=None) -> Optional[torch.Tensor]:
    """One device buffer large enough for the input-channel split of every (layer, shape); pools
    flags the layers called with the fused 2x2 max-pool."""
    pools = pools or [False] * len(layers)
    n = max([lay.workspace_bytes(s, p) for lay, s, p in zip(layers, x_shapes, pools)] + [0])
    if n == 0:
        return None
    return torch.empty(n // 4 + 4, dtype=torch.float32, device=device or "cuda")


def measure_fp32_peak(reps: int = 10) -> float:
    """Measured FP32 FMA peak of the current CUDA device in FLOP/s (pp_measure_fp32_peak)."""
    v = ctypes.c_double()
    _lib.check("pp_measure_fp32_peak", _lib.load().pp_measure_fp32_peak(int(reps), ctypes.byref(v)))
    return float(v.value)


def pp_maxpool2x2(x: torch.Tensor, out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """2x2/2 max-pool of a contiguous CUDA NCHW tensor via the library's kernel."""
    if not x.is_cuda or x.dtype not in _DT or not x.is_contiguous() or x.dim() != 4:
        raise ValueError("x must be a contiguous 4-d CUDA float32/float16 tensor (NCHW)")
    N, C, H, W = x.shape
    shape = (N, C, H // 2, W // 2)
    if out is None:
        out = torch.empty(shape, dtype=x.dtype, device=x.device)
    if tuple(out.shape) != shape or out.dtype != x.dtype or not out.is_contiguous():
        raise ValueError(f"out must be contiguous {shape} of x's dtype")
    _lib.check("pp_maxpool2x2", _lib.load().pp_maxpool2x2(
        ctypes.c_void_p(x.data_ptr()), _DT[x.dtype], N, C, H, W, ctypes.c_void_p(out.data_ptr()),
        _stream_ptr(stream, x.device)))
    return out
