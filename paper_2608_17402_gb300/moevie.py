"""Python binding of ``libmoevie.so`` -- argument marshalling only.

Every function below has the name of the C entry point it calls (``include/moevie.h``,
``include/moevie_testing.h``), takes torch CUDA tensors, passes their device
pointers and the current CUDA stream through ctypes, and raises
:class:`MoevieError` on a non-OK status.  All computation happens in the CUDA
library; there is no fallback of any kind: if the library is not built or no GPU
is present, the call fails.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libmoevie.so")
_lib = None

STATUS_NAMES = {0: "MOEVIE_OK", 1: "MOEVIE_ERR_INVALID_ARG", 2: "MOEVIE_ERR_UNSUPPORTED",
                3: "MOEVIE_ERR_WORKSPACE", 4: "MOEVIE_ERR_CUDA", 5: "MOEVIE_ERR_TIMEOUT",
                6: "MOEVIE_ERR_DEVICE"}
C_ENTRY_POINTS = ("moevie_status_string", "moevie_version", "moevie_workspace_size",
                  "moevie_workspace_init", "moevie_route", "moevie_permute", "moevie_permute_static",
                  "moevie_expert_ffn",
                  "moevie_shared_expert", "moevie_combine", "moevie_moe_forward", "moevie_moe_forward_host",
                  "moevie_get_device_status", "moevie_launch_count", "moevie_shared_groups",
                  "moevie_update_bias", "moevie_backward_workspace_size", "moevie_moe_backward",
                  "moevie_test_route_logits",
                  "moevie_test_fallback_count", "moevie_test_expert_hidden",
                  "moevie_test_moe_forward_events", "moevie_test_wait_timeout")


class MoevieError(RuntimeError):
    def __init__(self, fn, code):
        super().__init__(f"{fn} returned {STATUS_NAMES.get(code, code)}")
        self.code = code


class _Layer(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int64), ("E", ctypes.c_int64), ("k", ctypes.c_int64),
                ("h", ctypes.c_int64), ("h_s", ctypes.c_int64),
                ("W_r", ctypes.c_void_p), ("b", ctypes.c_void_p), ("W1", ctypes.c_void_p),
                ("W2", ctypes.c_void_p), ("Ws1", ctypes.c_void_p), ("Ws2", ctypes.c_void_p),
                ("lam", ctypes.c_float), ("W3", ctypes.c_void_p), ("Ws3", ctypes.c_void_p)]


class _Routing(ctypes.Structure):
    _fields_ = [("idx", ctypes.c_void_p), ("gate", ctypes.c_void_p), ("counts", ctypes.c_void_p),
                ("offsets", ctypes.c_void_p), ("perm", ctypes.c_void_p), ("inv", ctypes.c_void_p)]


def load():
    """Load the CUDA library (torch is imported first so both share one CUDA runtime)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is not built; run `python -c \"import __graft_entry__ as g; "
                          f"g.build()\"` first")
    lib = ctypes.CDLL(LIB_PATH)
    P, I64, SZ, F = ctypes.c_void_p, ctypes.c_int64, ctypes.c_size_t, ctypes.c_float
    sig = {
        "moevie_status_string": ([ctypes.c_int], ctypes.c_char_p),
        "moevie_version": ([], ctypes.c_int),
        "moevie_workspace_size": ([I64] * 6 + [P], ctypes.c_int),
        "moevie_workspace_init": ([P, SZ, P], ctypes.c_int),
        "moevie_route": ([P, P, P, I64, I64, I64, I64, P, P, P, SZ, P], ctypes.c_int),
        "moevie_permute": ([P, I64, I64, I64, P, P, P, P, P, SZ, P], ctypes.c_int),
        "moevie_permute_static": ([P, I64, I64, I64, P, P, P, P, P], ctypes.c_int),
        "moevie_expert_ffn": ([P, P, P, P, P, I64, I64, I64, I64, I64, P, P, SZ, P], ctypes.c_int),
        "moevie_shared_expert": ([P, P, P, I64, I64, I64, P, P, SZ, P], ctypes.c_int),
        "moevie_combine": ([P, P, P, P, F, I64, I64, I64, P, P], ctypes.c_int),
        "moevie_moe_forward": ([P, P, I64, P, P, P, SZ, P], ctypes.c_int),
        "moevie_moe_forward_host": ([P, P, I64, P, P, P, I64, P, SZ, P], ctypes.c_int),
        "moevie_get_device_status": ([P, P, P, P], ctypes.c_int),
        "moevie_launch_count": ([], ctypes.c_uint64),
        "moevie_shared_groups": ([I64] * 6, ctypes.c_int64),
        "moevie_update_bias": ([P, I64, F, ctypes.c_int, P, P, SZ, P], ctypes.c_int),
        "moevie_backward_workspace_size": ([I64] * 6 + [ctypes.c_int, P], ctypes.c_int),
        "moevie_moe_backward": ([P, P, P, I64, P, P, P, P, P, P, P, P, P, P, SZ, P], ctypes.c_int),
        "moevie_test_route_logits": ([P, P, I64, I64, I64, P, P, SZ, P], ctypes.c_int),
        "moevie_test_fallback_count": ([P, P, P], ctypes.c_int),
        "moevie_test_expert_hidden": ([P, P, P, P, I64, I64, I64, I64, I64, P, P, SZ, P],
                                      ctypes.c_int),
        "moevie_test_moe_forward_events": ([P, P, I64, P, P, SZ, P, P, ctypes.c_int], ctypes.c_int),
        "moevie_test_wait_timeout": ([P, SZ, ctypes.c_uint64, P], ctypes.c_int),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    _lib = lib
    return lib


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _call(name, *args):
    rc = getattr(load(), name)(*args)
    if rc != 0:
        raise MoevieError(name, rc)


def _want(t, dtype, name):
    if not (t.is_cuda and t.dtype == dtype and t.is_contiguous()):
        raise ValueError(f"{name}: expected a contiguous CUDA {dtype} tensor, got "
                         f"{t.dtype} on {t.device} (contiguous={t.is_contiguous()})")
    return t


def row_ld(h: int) -> int:
    """Row stride (elements) of W1, W3, Ws1, Ws3 and the hidden activations when a
    row holds h values: rows start 16 bytes apart (h rounded up to a multiple of 8)."""
    return (h + 7) // 8 * 8


def _rows_ok(t) -> bool:
    """t [..., h] has row stride row_ld(h) and is otherwise packed."""
    want = 1
    for i in range(t.dim() - 1, -1, -1):
        if t.shape[i] != 1 and t.stride(i) != want:
            return False
        want *= row_ld(t.shape[i]) if i == t.dim() - 1 else t.shape[i]
    return True


def moevie_pad_rows(w: torch.Tensor) -> torch.Tensor:
    """``w`` [..., h] laid out as the entry points take W1, W3, Ws1 and Ws3 (row
    stride ``row_ld(h)``, the pad never read): ``w`` itself when it already is, else
    a copy into a zero-padded buffer, returned as its [..., h] view."""
    if _rows_ok(w):
        return w
    h = w.shape[-1]
    buf = torch.zeros(*w.shape[:-1], row_ld(h), dtype=w.dtype, device=w.device)
    buf[..., :h].copy_(w)
    return buf[..., :h]


def _want_rows(t, dtype, name):
    if not (t.is_cuda and t.dtype == dtype and _rows_ok(t)):
        raise ValueError(f"{name}: expected a CUDA {dtype} tensor [..., h] with row stride "
                         f"row_ld(h) (see moevie_pad_rows), got {t.dtype} on {t.device} with "
                         f"shape {tuple(t.shape)} and strides {t.stride()}")
    return t


# ------------------------------------------------------------------ workspace

def moevie_workspace_size(T_max, d, E, k, h, h_s=0) -> int:
    out = ctypes.c_size_t(0)
    _call("moevie_workspace_size", T_max, d, E, k, h, h_s, ctypes.byref(out))
    return out.value


class Workspace:
    """Caller-owned device scratch for the layer (sized for up to ``T_max`` tokens)."""

    def __init__(self, T_max, d, E, k, h, h_s=0, device="cuda", stream=None):
        self.dims = (T_max, d, E, k, h, h_s)
        self.nbytes = moevie_workspace_size(T_max, d, E, k, h, h_s)
        self.buf = torch.empty(self.nbytes, dtype=torch.uint8, device=device)
        moevie_workspace_init(self, stream)

    @property
    def ptr(self):
        return ctypes.c_void_p(self.buf.data_ptr())


def moevie_workspace_init(ws: Workspace, stream=None):
    _call("moevie_workspace_init", ws.ptr, ws.nbytes, _stream(stream))


def moevie_get_device_status(ws: Workspace, stream=None):
    """Synchronises the stream; returns ``(code, [code, site, a, b])``."""
    code = ctypes.c_int(0)
    detail = (ctypes.c_int32 * 4)()
    _call("moevie_get_device_status", ws.ptr, _stream(stream), ctypes.byref(code), detail)
    return code.value, list(detail)


# ----------------------------------------------------------------- the stages

def moevie_route(x, W_r, b, k, ws: Workspace, idx=None, gate=None, stream=None):
    _want(x, torch.bfloat16, "x")
    _want(W_r, torch.float32, "W_r")
    _want(b, torch.float32, "b")
    T, d = x.shape
    E = W_r.shape[1]
    idx = idx if idx is not None else torch.empty((T, k), dtype=torch.int32, device=x.device)
    gate = gate if gate is not None else torch.empty((T, k), dtype=torch.float32, device=x.device)
    _call("moevie_route", _p(x), _p(W_r), _p(b), T, d, E, k, _p(idx), _p(gate), ws.ptr, ws.nbytes,
          _stream(stream))
    return idx, gate


def moevie_permute(idx, E, ws: Workspace, stream=None):
    _want(idx, torch.int32, "idx")
    T, k = idx.shape
    dev = idx.device
    counts = torch.empty(E, dtype=torch.int32, device=dev)
    offsets = torch.empty(E + 1, dtype=torch.int32, device=dev)
    perm = torch.empty(T * k, dtype=torch.int32, device=dev)
    inv = torch.empty(T * k, dtype=torch.int32, device=dev)
    _call("moevie_permute", _p(idx), T, k, E, _p(counts), _p(offsets), _p(perm), _p(inv), ws.ptr,
          ws.nbytes, _stream(stream))
    return counts, offsets, perm, inv


def moevie_permute_static(idx, E, out=None, stream=None):
    """moevie_permute without a workspace: the library's fixed device scratch is used
    (T * k <= 2^20).  Calls whose GPU work overlaps race on that scratch.  ``out``: an
    optional tuple of preallocated (counts [E], offsets [E + 1], perm [T*k], inv [T*k])
    int32 tensors, so that the call itself allocates nothing."""
    _want(idx, torch.int32, "idx")
    T, k = idx.shape
    dev = idx.device
    if out is not None:
        counts, offsets, perm, inv = (_want(t, torch.int32, n)
                                      for t, n in zip(out, ("counts", "offsets", "perm", "inv")))
        if counts.numel() != E or offsets.numel() != E + 1 or perm.numel() < T * k or inv.numel() < T * k:
            raise ValueError("moevie_permute_static: output tensors of the wrong size")
    else:
        counts = torch.empty(E, dtype=torch.int32, device=dev)
        offsets = torch.empty(E + 1, dtype=torch.int32, device=dev)
        perm = torch.empty(T * k, dtype=torch.int32, device=dev)
        inv = torch.empty(T * k, dtype=torch.int32, device=dev)
    _call("moevie_permute_static", _p(idx), T, k, E, _p(counts), _p(offsets), _p(perm), _p(inv),
          _stream(stream))
    return counts, offsets, perm, inv


def moevie_expert_ffn(x, perm, offsets, W1, W2, k, ws: Workspace, out_rows=None, stream=None):
    _want(x, torch.bfloat16, "x")
    _want_rows(W1, torch.bfloat16, "W1")
    _want(W2, torch.bfloat16, "W2")
    T, d = x.shape
    E, _, h = W1.shape
    out_rows = out_rows if out_rows is not None else torch.empty((T * k, d), dtype=torch.bfloat16,
                                                                 device=x.device)
    _call("moevie_expert_ffn", _p(x), _p(perm), _p(offsets), _p(W1), _p(W2), T, d, h, E, k,
          _p(out_rows), ws.ptr, ws.nbytes, _stream(stream))
    return out_rows


def moevie_shared_expert(x, Ws1, Ws2, ws: Workspace, out=None, stream=None):
    _want(x, torch.bfloat16, "x")
    _want_rows(Ws1, torch.bfloat16, "Ws1")
    _want(Ws2, torch.bfloat16, "Ws2")
    T, d = x.shape
    hs = Ws1.shape[1]
    out = out if out is not None else torch.empty((T, d), dtype=torch.bfloat16, device=x.device)
    _call("moevie_shared_expert", _p(x), _p(Ws1), _p(Ws2), T, d, hs, _p(out), ws.ptr, ws.nbytes,
          _stream(stream))
    return out


def moevie_combine(out_rows, inv, gate, k, shared_out=None, lam=1.0, y=None, stream=None):
    _want(out_rows, torch.bfloat16, "out_rows")
    T = gate.shape[0]
    d = out_rows.shape[1]
    y = y if y is not None else torch.empty((T, d), dtype=torch.bfloat16, device=out_rows.device)
    _call("moevie_combine", _p(out_rows), _p(inv), _p(gate), _p(shared_out), float(lam), T, k, d,
          _p(y), _stream(stream))
    return y


@dataclass
class LayerWeights:
    """Device weights of one layer (bf16 unless noted)."""
    W_r: torch.Tensor           # fp32 [d, E]
    b: torch.Tensor             # fp32 [E]
    W1: torch.Tensor            # [E, d, h], row stride row_ld(h) (moevie_pad_rows)
    W2: torch.Tensor            # [E, h, d]
    k: int
    Ws1: torch.Tensor | None = None   # [d, h_s], row stride row_ld(h_s)
    Ws2: torch.Tensor | None = None   # [h_s, d]
    lam: float = 1.0
    W3: torch.Tensor | None = None    # [E, d, h] as W1: SwiGLU experts (W1 gate, W3 up); None: GELU
    Ws3: torch.Tensor | None = None   # [d, h_s] as Ws1: with W3, the SwiGLU shared expert's up

    @property
    def dims(self):
        d, E = self.W_r.shape
        h = self.W1.shape[2]
        hs = 0 if self.Ws1 is None else self.Ws1.shape[1]
        return d, E, self.k, h, hs

    def c_struct(self) -> _Layer:
        d, E, k, h, hs = self.dims
        for name in ("W1", "W3", "Ws1", "Ws3"):
            if getattr(self, name) is not None:
                _want_rows(getattr(self, name), torch.bfloat16, name)
        return _Layer(d, E, k, h, hs, self.W_r.data_ptr(), self.b.data_ptr(), self.W1.data_ptr(),
                      self.W2.data_ptr(), 0 if self.Ws1 is None else self.Ws1.data_ptr(),
                      0 if self.Ws2 is None else self.Ws2.data_ptr(), float(self.lam),
                      0 if self.W3 is None else self.W3.data_ptr(),
                      0 if self.Ws3 is None else self.Ws3.data_ptr())


def moevie_moe_forward(layer: LayerWeights, x, ws: Workspace, y=None, routing=False, stream=None):
    """The fused layer forward.  With ``routing=True`` also returns a dict of the
    routing by-products (idx, gate, counts, offsets, perm, inv)."""
    _want(x, torch.bfloat16, "x")
    T, d = x.shape
    _, E, k, _, _ = layer.dims
    dev = x.device
    y = y if y is not None else torch.empty((T, d), dtype=torch.bfloat16, device=dev)
    rt = None
    rstruct = None
    if routing:
        rt = {"idx": torch.empty((T, k), dtype=torch.int32, device=dev),
              "gate": torch.empty((T, k), dtype=torch.float32, device=dev),
              "counts": torch.empty(E, dtype=torch.int32, device=dev),
              "offsets": torch.empty(E + 1, dtype=torch.int32, device=dev),
              "perm": torch.empty(T * k, dtype=torch.int32, device=dev),
              "inv": torch.empty(T * k, dtype=torch.int32, device=dev)}
        rstruct = _Routing(*(rt[n].data_ptr() for n in ("idx", "gate", "counts", "offsets", "perm",
                                                         "inv")))
    L = layer.c_struct()
    _call("moevie_moe_forward", ctypes.byref(L), _p(x), T, _p(y),
          ctypes.byref(rstruct) if rstruct is not None else None, ws.ptr, ws.nbytes,
          _stream(stream))
    return (y, rt) if routing else y


HOST_MAX_CHUNKS = 16   # MOEVIE_HOST_MAX_CHUNKS


def host_chunks(T: int) -> int:
    """A chunk count for moevie_moe_forward_host: pieces of at least 32768 tokens (each
    piece is a whole layer forward, and smaller ones lose more to weight reads and partial
    tiles than the overlap wins), at most 16.  Measured on GB300 with the half-size first
    and last pieces: T = 65536 in 2 chunks 2.90 ms against 4.20 ms in one and 3.02 ms in
    4; T = 32768 in 2 chunks 1.37 ms against 1.92 ms; T = 8192 best in one."""
    return 1 if T < 32768 else max(2, min(HOST_MAX_CHUNKS, T // 32768))


def moevie_moe_forward_host(layer: LayerWeights, x_host, y_host, x_dev, y_dev, ws: Workspace, chunks: int,
                            stream=None):
    """The layer from host to host memory with the copies overlapped (moevie_moe_forward_host):
    x_host, y_host CPU bf16 [T, d] (pinned for overlap); x_dev, y_dev CUDA bf16 [T, d] scratch;
    ws a Workspace for ceil(T / chunks) tokens.  Asynchronous on `stream`, which completes
    after the last row of y_host is written."""
    _want(x_dev, torch.bfloat16, "x_dev")
    _want(y_dev, torch.bfloat16, "y_dev")
    for name, t in (("x_host", x_host), ("y_host", y_host)):
        if t.device.type != "cpu" or t.dtype != torch.bfloat16 or not t.is_contiguous():
            raise ValueError(f"{name}: expected a contiguous CPU bfloat16 tensor")
    T, d = x_host.shape
    if tuple(y_host.shape) != (T, d) or tuple(x_dev.shape) != (T, d) or tuple(y_dev.shape) != (T, d):
        raise ValueError("x_host, y_host, x_dev and y_dev must all be [T, d]")
    L = layer.c_struct()
    _call("moevie_moe_forward_host", ctypes.byref(L), ctypes.c_void_p(x_host.data_ptr()), T,
          ctypes.c_void_p(y_host.data_ptr()), _p(x_dev), _p(y_dev), int(chunks), ws.ptr, ws.nbytes,
          _stream(stream))
    return y_host


def moevie_backward_workspace_size(T_max, d, E, k, h, h_s=0, swiglu=False) -> int:
    out = ctypes.c_size_t(0)
    _call("moevie_backward_workspace_size", T_max, d, E, k, h, h_s, int(bool(swiglu)), ctypes.byref(out))
    return out.value


class BackwardWorkspace(Workspace):
    """Caller-owned device scratch of moevie_moe_backward (up to ``T_max`` tokens;
    ``h_s`` the shared expert's width, 0 for none; ``swiglu`` for SwiGLU experts)."""

    def __init__(self, T_max, d, E, k, h, h_s=0, swiglu=False, device="cuda", stream=None):
        self.dims = (T_max, d, E, k, h, h_s, swiglu)
        self.nbytes = moevie_backward_workspace_size(T_max, d, E, k, h, h_s, swiglu)
        self.buf = torch.empty(self.nbytes, dtype=torch.uint8, device=device)
        moevie_workspace_init(self, stream)


def moevie_moe_backward(layer: LayerWeights, x, dy, idx, ws: "BackwardWorkspace", stream=None):
    """Gradients of sum(dy * y) with the selection idx held fixed (GELU or SwiGLU
    experts, with or without a shared expert).  Returns a dict of fp32 tensors: dx [T, d],
    dW_r [d, E], dW1 [E, d, h] (a view of rows row_ld(h) apart), dW2 [E, h, d], dW3 (as
    dW1) for SwiGLU experts, and with a shared expert dWs1 [d, h_s] (a view of rows
    row_ld(h_s) apart), dWs2 [h_s, d] and, for SwiGLU, dWs3 (as dWs1)."""
    _want(x, torch.bfloat16, "x")
    _want(dy, torch.bfloat16, "dy")
    _want(idx, torch.int32, "idx")
    T, d = x.shape
    _, E, k, h, hs = layer.dims
    dev = x.device
    out = {"dx": torch.empty((T, d), dtype=torch.float32, device=dev),
           "dW_r": torch.empty((d, E), dtype=torch.float32, device=dev),
           "dW1": torch.empty((E, d, row_ld(h)), dtype=torch.float32, device=dev),
           "dW2": torch.empty((E, h, d), dtype=torch.float32, device=dev)}
    if layer.W3 is not None:
        out["dW3"] = torch.empty((E, d, row_ld(h)), dtype=torch.float32, device=dev)
    if hs > 0:
        out["dWs1"] = torch.empty((d, row_ld(hs)), dtype=torch.float32, device=dev)
        out["dWs2"] = torch.empty((hs, d), dtype=torch.float32, device=dev)
        if layer.W3 is not None:
            out["dWs3"] = torch.empty((d, row_ld(hs)), dtype=torch.float32, device=dev)
    L = layer.c_struct()
    _call("moevie_moe_backward", ctypes.byref(L), _p(x), _p(dy), T, _p(idx), _p(out["dx"]), _p(out["dW_r"]),
          _p(out["dW1"]), _p(out["dW2"]), _p(out.get("dW3")), _p(out.get("dWs1")), _p(out.get("dWs2")),
          _p(out.get("dWs3")), ws.ptr, ws.nbytes, _stream(stream))
    out["dW1"] = out["dW1"][..., :h]
    for name, w in (("dW3", h), ("dWs1", hs), ("dWs3", hs)):
        if name in out:
            out[name] = out[name][..., :w]
    return out


def moevie_launch_count() -> int:
    return int(load().moevie_launch_count())


def moevie_update_bias(counts, b, alpha, ws: "Workspace", rule="zscore", stream=None):
    """Loss-free bias update in place on b (fp32 [E]) from counts (int32 [E]): z-score
    rule (Eq. 9) or sign rule (Eq. 8)."""
    _want(counts, torch.int32, "counts")
    _want(b, torch.float32, "b")
    r = {"zscore": 0, "sign": 1}[rule]
    _call("moevie_update_bias", _p(counts), counts.numel(), float(alpha), r, _p(b), ws.ptr, ws.nbytes,
          _stream(stream))
    return b


def moevie_shared_groups(T, d, E, k, h, h_s) -> int:
    """Always-on groups that carry the shared expert inside the routed GEMMs (0: own GEMMs)."""
    return int(load().moevie_shared_groups(T, d, E, k, h, h_s))


# ----------------------------------------------------------------- test hooks

FORWARD_STAGES = ("route", "permute", "y_init", "up_gemm", "down_gemm", "finalize")


def moevie_test_moe_forward_events(layer: LayerWeights, x, ws: Workspace, events, y=None,
                                   stream=None):
    """Forward that records the 7 stage-boundary events (torch.cuda.Event objects,
    already recorded once so that their CUDA handles exist)."""
    T, d = x.shape
    y = y if y is not None else torch.empty((T, d), dtype=torch.bfloat16, device=x.device)
    arr = (ctypes.c_void_p * 7)(*(ctypes.c_void_p(e.cuda_event) for e in events))
    L = layer.c_struct()
    _call("moevie_test_moe_forward_events", ctypes.byref(L), _p(x), T, _p(y), ws.ptr, ws.nbytes,
          _stream(stream), arr, 7)
    return y


def moevie_test_route_logits(x, W_r, ws: Workspace, stream=None):
    """Fast-path logits [T, E] (the library writes E rounded up to 32 columns)."""
    T, d = x.shape
    E = W_r.shape[1]
    E32 = (E + 31) // 32 * 32
    s = torch.empty((T, E32), dtype=torch.float32, device=x.device)
    _call("moevie_test_route_logits", _p(x), _p(W_r), T, d, E, _p(s), ws.ptr, ws.nbytes,
          _stream(stream))
    return s[:, :E]


def moevie_test_fallback_count(ws: Workspace, stream=None) -> int:
    out = ctypes.c_int32(0)
    _call("moevie_test_fallback_count", ws.ptr, _stream(stream), ctypes.byref(out))
    return out.value


def moevie_test_expert_hidden(x, perm, offsets, W1, k, ws: Workspace, stream=None):
    T, d = x.shape
    _want_rows(W1, torch.bfloat16, "W1")
    E, _, h = W1.shape
    hidden = torch.empty((T * k, row_ld(h)), dtype=torch.bfloat16, device=x.device)
    _call("moevie_test_expert_hidden", _p(x), _p(perm), _p(offsets), _p(W1), T, d, h, E, k,
          _p(hidden), ws.ptr, ws.nbytes, _stream(stream))
    return hidden[:, :h]


def moevie_test_wait_timeout(ws: Workspace, limit_ns: int, stream=None):
    _call("moevie_test_wait_timeout", ws.ptr, ws.nbytes, ctypes.c_uint64(limit_ns), _stream(stream))
