"""ctypes binding of libclearmoe.so, one Python function per C entry point (same names).

Argument marshalling only: tensors become device pointers, torch's current stream becomes the
cudaStream_t, non-zero status codes become ClearMoEError. Every step of the layer runs in the
library's CUDA kernels; there is no Python or CPU fallback. The C declarations, with argument
meaning, layout, ownership and errors, are in include/clearmoe.h.
"""
from __future__ import annotations

import ctypes
import pathlib

_LIB_PATH = pathlib.Path(__file__).resolve().parent / "libclearmoe.so"
_lib = None

OK, EINVAL, EUNSUPPORTED, ECUDA, ENOMEM, ETIMEOUT = 0, -1, -2, -3, -4, -5
F32, BF16 = 0, 1


class ClearMoEError(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"{where}: {clearmoe_strerror(code)} ({code})")
        self.code = code


class clearmoe_layer_desc(ctypes.Structure):
    _fields_ = [("max_tokens", ctypes.c_int64), ("d", ctypes.c_int32), ("hidden", ctypes.c_int32),
                ("max_E", ctypes.c_int32), ("max_r", ctypes.c_int32), ("dtype", ctypes.c_int32)]


class clearmoe_router(ctypes.Structure):
    _fields_ = [("W", ctypes.c_void_p), ("b", ctypes.c_void_p)]


class clearmoe_mlp_router(ctypes.Structure):
    _fields_ = [("W_in", ctypes.c_void_p), ("b_in", ctypes.c_void_p), ("W_out", ctypes.c_void_p),
                ("b_out", ctypes.c_void_p), ("hidden", ctypes.c_int32), ("act", ctypes.c_int32)]


class clearmoe_ffn_options(ctypes.Structure):
    _fields_ = [("b2", ctypes.c_void_p), ("cls_stride", ctypes.c_int64), ("W2", ctypes.c_void_p),
                ("mlp_router", ctypes.POINTER(clearmoe_mlp_router)), ("input_layernorm", ctypes.c_int32),
                ("router_in_fc1", ctypes.c_int32)]


ACT_RELU, ACT_GELU = 0, 1


def mlp_router(W_in, b_in, W_out, b_out, act: str = "relu") -> clearmoe_mlp_router:
    """The MLP router's weights as the C struct (act: "relu" or "gelu")."""
    return clearmoe_mlp_router(_ptr(W_in), _ptr(b_in), _ptr(W_out), _ptr(b_out), W_in.shape[0],
                               {"relu": ACT_RELU, "gelu": ACT_GELU}[act])


_P, _I64, _I32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
_SIGS = {
    "clearmoe_layer_create": [ctypes.POINTER(clearmoe_layer_desc), ctypes.POINTER(ctypes.c_void_p)],
    "clearmoe_layer_destroy": [_P],
    "clearmoe_route": [_P, _P, _I64, ctypes.POINTER(clearmoe_router), _I32, _P],
    "clearmoe_route_mlp": [_P, _P, _I64, ctypes.POINTER(clearmoe_mlp_router), _I32, _P],
    "clearmoe_ffn_forward": [_P, _P, _I64, _P, _P, _P, _P, _P, ctypes.POINTER(ctypes.c_void_p),
                             ctypes.POINTER(clearmoe_router), _I32, _I32, _P, _P],
    "clearmoe_ffn_forward_ex": [_P, _P, _I64, _P, _P, _P, _P, _P, ctypes.POINTER(ctypes.c_void_p),
                                ctypes.POINTER(clearmoe_router), _I32, _I32,
                                ctypes.POINTER(clearmoe_ffn_options), _P, _P],
    "clearmoe_materialize_basis": [_P, _P, _P, _P, _I32, _P, _P],
    "clearmoe_ffn_forward_folded_ex": [_P, _P, _I64, _P, _P, ctypes.POINTER(ctypes.c_void_p),
                                       ctypes.POINTER(clearmoe_router), _I32,
                                       ctypes.POINTER(clearmoe_ffn_options), _P, _P],
    "clearmoe_ffn_forward_materialized_ex": [_P, _P, _I64, _P, _P, _P, ctypes.POINTER(ctypes.c_void_p),
                                             ctypes.POINTER(clearmoe_router), _I32,
                                             ctypes.POINTER(clearmoe_ffn_options), _P, _P],
    "clearmoe_ffn_forward_materialized": [_P, _P, _I64, _P, _P, _P, ctypes.POINTER(ctypes.c_void_p),
                                          ctypes.POINTER(clearmoe_router), _I32, _P, _P],
    "clearmoe_ffn_forward_scaled": [_P, _P, _I64, _P, _P, _P, _P, _P, _P, _P,
                                    ctypes.POINTER(clearmoe_router), _I32, _I32, _P, _P],
    "clearmoe_dense_ffn_forward": [_P, _P, _I64, _P, _P, _P, _P, _P],
    "clearmoe_dense_ffn_forward_ex": [_P, _P, _I64, _P, _P, _P, _P, _P, _P],
    "clearmoe_dense_ffn_forward_opt": [_P, _P, _I64, _P, _P, _P, ctypes.POINTER(clearmoe_ffn_options), _P, _P],
    "clearmoe_layer_norm": [_P, _P, _I64, _P, _P],
    "clearmoe_get_routing": [_P, _P, _P, _P, _P, _P],
    "clearmoe_layer_status": [_P],
    "clearmoe_debug_set_wait": [_P, _I64, _I32],
    "clearmoe_set_profile_events": [_P, ctypes.POINTER(ctypes.c_void_p), _I32],
    "clearmoe_fold_basis": [_P, _P, _P, _P, ctypes.POINTER(ctypes.c_void_p), _I32, _I32,
                            ctypes.POINTER(ctypes.c_void_p), _P],
    "clearmoe_ffn_forward_folded": [_P, _P, _I64, _P, _P, ctypes.POINTER(ctypes.c_void_p),
                                    ctypes.POINTER(clearmoe_router), _I32, _P, _P],
    "clearmoe_route_noalloc": [_P, _I64, _I32, _I32, ctypes.POINTER(clearmoe_router), _I32, _P, _P,
                               _P, _P, _P, _P],
    "clearmoe_strerror": [ctypes.c_int],
    "clearmoe_version": [],
}


def lib() -> ctypes.CDLL:
    """Loads libclearmoe.so (built in-tree). Raises if it is missing: there is no fallback."""
    global _lib
    if _lib is None:
        if not _LIB_PATH.exists():
            raise RuntimeError(f"{_LIB_PATH} is not built; run paper_2606_28516_gb300.build.build()")
        try:
            import torch  # noqa: F401  (loads the CUDA runtime the library links against)
        except ImportError:
            pass
        L = ctypes.CDLL(str(_LIB_PATH))
        for name, args in _SIGS.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = ctypes.c_char_p if name == "clearmoe_strerror" else ctypes.c_int
        _lib = L
    return _lib


def _check(code: int, where: str) -> None:
    if code != OK:
        raise ClearMoEError(code, where)


def _ptr(t) -> int | None:
    if t is None:
        return None
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("tensors passed to libclearmoe must be contiguous CUDA tensors")
    return t.data_ptr()


def _stream(stream) -> int | None:
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


def clearmoe_strerror(code: int) -> str:
    return lib().clearmoe_strerror(code).decode()


def clearmoe_version() -> int:
    return lib().clearmoe_version()


def clearmoe_layer_create(max_tokens: int, d: int, hidden: int, max_E: int, max_r: int,
                          dtype: int) -> int:
    desc = clearmoe_layer_desc(max_tokens, d, hidden, max_E, max_r, dtype)
    h = ctypes.c_void_p()
    _check(lib().clearmoe_layer_create(ctypes.byref(desc), ctypes.byref(h)), "clearmoe_layer_create")
    return h.value


def clearmoe_layer_destroy(layer: int) -> None:
    _check(lib().clearmoe_layer_destroy(layer), "clearmoe_layer_destroy")


def _router(Wg, bg) -> clearmoe_router:
    return clearmoe_router(_ptr(Wg), _ptr(bg))


def clearmoe_route(layer: int, x, Wg, bg, stream=None) -> None:
    r = _router(Wg, bg)
    _check(lib().clearmoe_route(layer, _ptr(x), x.shape[0], ctypes.byref(r), Wg.shape[0],
                                _stream(stream)), "clearmoe_route")


def clearmoe_route_mlp(layer: int, x, mlp: clearmoe_mlp_router, E: int, stream=None) -> None:
    _check(lib().clearmoe_route_mlp(layer, _ptr(x), x.shape[0], ctypes.byref(mlp), E, _stream(stream)),
           "clearmoe_route_mlp")


def clearmoe_ffn_forward(layer: int, x, W1, b1, U_r, S_r, Vh_r, residual_e, Wg, bg, out,
                         stream=None) -> None:
    """residual_e: a sequence of E [d x H] tensors, or one [E x d x H] tensor."""
    E = Wg.shape[0]
    res = (ctypes.c_void_p * E)(*[_ptr(residual_e[e]) for e in range(E)])
    r = _router(Wg, bg)
    _check(lib().clearmoe_ffn_forward(layer, _ptr(x), x.shape[0], _ptr(W1), _ptr(b1), _ptr(U_r),
                                      _ptr(S_r), _ptr(Vh_r), res, ctypes.byref(r), E,
                                      S_r.shape[0], _ptr(out), _stream(stream)),
           "clearmoe_ffn_forward")


def clearmoe_ffn_forward_ex(layer: int, x, W1, b1, U_r, S_r, Vh_r, residual_e, Wg, bg, out,
                            b2=None, W2=None, cls_stride: int = 0, mlp: clearmoe_mlp_router | None = None,
                            E: int | None = None, input_layernorm: bool = False, router_in_fc1: bool = False,
                            stream=None) -> None:
    """clearmoe_ffn_forward with fc2's bias b2, class tokens (every cls_stride-th token from token 0)
    on the dense path W2, the MLP router `mlp` (then Wg, bg may be None and E is given),
    input_layernorm (x is the un-normalised stream y; the layer's input is LN(y)), and
    router_in_fc1 (the linear router's logits computed inside fc1)."""
    E = Wg.shape[0] if E is None else E
    res = (ctypes.c_void_p * E)(*[_ptr(residual_e[e]) for e in range(E)])
    r = _router(Wg, bg) if Wg is not None else None
    opt = _options(b2, W2, cls_stride, mlp, input_layernorm, router_in_fc1)
    _check(lib().clearmoe_ffn_forward_ex(layer, _ptr(x), x.shape[0], _ptr(W1), _ptr(b1), _ptr(U_r),
                                         _ptr(S_r), _ptr(Vh_r), res, ctypes.byref(r) if r else None, E,
                                         S_r.shape[0], ctypes.byref(opt), _ptr(out),
                                         _stream(stream)), "clearmoe_ffn_forward_ex")


def clearmoe_fold_basis(layer: int, U_r, S_r, Vh_r, residual_e, W_comb, stream=None) -> None:
    """residual_e, W_comb: sequences of E [d x H] tensors, or [E x d x H] tensors."""
    E = len(residual_e)
    res = (ctypes.c_void_p * E)(*[_ptr(residual_e[e]) for e in range(E)])
    comb = (ctypes.c_void_p * E)(*[_ptr(W_comb[e]) for e in range(E)])
    _check(lib().clearmoe_fold_basis(layer, _ptr(U_r), _ptr(S_r), _ptr(Vh_r), res, E, S_r.shape[0],
                                     comb, _stream(stream)), "clearmoe_fold_basis")


def clearmoe_ffn_forward_folded(layer: int, x, W1, b1, W_comb, Wg, bg, out, stream=None) -> None:
    E = Wg.shape[0]
    comb = (ctypes.c_void_p * E)(*[_ptr(W_comb[e]) for e in range(E)])
    r = _router(Wg, bg)
    _check(lib().clearmoe_ffn_forward_folded(layer, _ptr(x), x.shape[0], _ptr(W1), _ptr(b1), comb,
                                             ctypes.byref(r), E, _ptr(out), _stream(stream)),
           "clearmoe_ffn_forward_folded")


def clearmoe_materialize_basis(layer: int, U_r, S_r, Vh_r, W_sh, stream=None) -> None:
    _check(lib().clearmoe_materialize_basis(layer, _ptr(U_r), _ptr(S_r), _ptr(Vh_r), S_r.shape[0],
                                            _ptr(W_sh), _stream(stream)), "clearmoe_materialize_basis")


def clearmoe_ffn_forward_materialized(layer: int, x, W1, b1, W_sh, residual_e, Wg, bg, out,
                                      stream=None) -> None:
    E = Wg.shape[0]
    res = (ctypes.c_void_p * E)(*[_ptr(residual_e[e]) for e in range(E)])
    r = _router(Wg, bg)
    _check(lib().clearmoe_ffn_forward_materialized(layer, _ptr(x), x.shape[0], _ptr(W1), _ptr(b1),
                                                   _ptr(W_sh), res, ctypes.byref(r), E, _ptr(out),
                                                   _stream(stream)), "clearmoe_ffn_forward_materialized")


def clearmoe_ffn_forward_scaled(layer: int, x, W1, b1, U_r, S_r, Vh_r, R, s_e, Wg, bg, out,
                                stream=None) -> None:
    r = _router(Wg, bg)
    _check(lib().clearmoe_ffn_forward_scaled(layer, _ptr(x), x.shape[0], _ptr(W1), _ptr(b1), _ptr(U_r),
                                             _ptr(S_r), _ptr(Vh_r), _ptr(R), _ptr(s_e), ctypes.byref(r),
                                             Wg.shape[0], S_r.shape[0], _ptr(out), _stream(stream)),
           "clearmoe_ffn_forward_scaled")


def _options(b2, W2, cls_stride, mlp, input_layernorm=False, router_in_fc1=False):
    return clearmoe_ffn_options(_ptr(b2), int(cls_stride), _ptr(W2),
                                ctypes.pointer(mlp) if mlp is not None else None, int(bool(input_layernorm)),
                                int(bool(router_in_fc1)))


def clearmoe_ffn_forward_folded_ex(layer: int, x, W1, b1, W_comb, Wg, bg, out, b2=None, W2=None,
                                   cls_stride: int = 0, mlp: clearmoe_mlp_router | None = None,
                                   E: int | None = None, input_layernorm: bool = False,
                                   router_in_fc1: bool = False, stream=None) -> None:
    E = Wg.shape[0] if E is None else E
    comb = (ctypes.c_void_p * E)(*[_ptr(W_comb[e]) for e in range(E)])
    r = _router(Wg, bg) if Wg is not None else None
    opt = _options(b2, W2, cls_stride, mlp, input_layernorm, router_in_fc1)
    _check(lib().clearmoe_ffn_forward_folded_ex(layer, _ptr(x), x.shape[0], _ptr(W1), _ptr(b1), comb,
                                                ctypes.byref(r) if r else None, E, ctypes.byref(opt),
                                                _ptr(out), _stream(stream)), "clearmoe_ffn_forward_folded_ex")


def clearmoe_ffn_forward_materialized_ex(layer: int, x, W1, b1, W_sh, residual_e, Wg, bg, out, b2=None,
                                         W2=None, cls_stride: int = 0,
                                         mlp: clearmoe_mlp_router | None = None, E: int | None = None,
                                         input_layernorm: bool = False, router_in_fc1: bool = False,
                                         stream=None) -> None:
    E = Wg.shape[0] if E is None else E
    res = (ctypes.c_void_p * E)(*[_ptr(residual_e[e]) for e in range(E)])
    r = _router(Wg, bg) if Wg is not None else None
    opt = _options(b2, W2, cls_stride, mlp, input_layernorm, router_in_fc1)
    _check(lib().clearmoe_ffn_forward_materialized_ex(layer, _ptr(x), x.shape[0], _ptr(W1), _ptr(b1),
                                                      _ptr(W_sh), res, ctypes.byref(r) if r else None, E,
                                                      ctypes.byref(opt), _ptr(out), _stream(stream)),
           "clearmoe_ffn_forward_materialized_ex")


def clearmoe_dense_ffn_forward(layer: int, x, W1, b1, W2, out, stream=None) -> None:
    _check(lib().clearmoe_dense_ffn_forward(layer, _ptr(x), x.shape[0], _ptr(W1), _ptr(b1),
                                            _ptr(W2), _ptr(out), _stream(stream)),
           "clearmoe_dense_ffn_forward")


def clearmoe_dense_ffn_forward_ex(layer: int, x, W1, b1, W2, b2, out, stream=None) -> None:
    _check(lib().clearmoe_dense_ffn_forward_ex(layer, _ptr(x), x.shape[0], _ptr(W1), _ptr(b1),
                                               _ptr(W2), _ptr(b2), _ptr(out), _stream(stream)),
           "clearmoe_dense_ffn_forward_ex")


def clearmoe_dense_ffn_forward_opt(layer: int, x, W1, b1, W2, out, b2=None, input_layernorm: bool = False,
                                   stream=None) -> None:
    """The dense FFN with fc2's bias b2 and input_layernorm (x is y; the input is LN(y))."""
    opt = _options(b2, None, 0, None, input_layernorm)
    _check(lib().clearmoe_dense_ffn_forward_opt(layer, _ptr(x), x.shape[0], _ptr(W1), _ptr(b1), _ptr(W2),
                                                ctypes.byref(opt), _ptr(out), _stream(stream)),
           "clearmoe_dense_ffn_forward_opt")


def clearmoe_layer_norm(layer: int, y, x_out, stream=None) -> None:
    _check(lib().clearmoe_layer_norm(layer, _ptr(y), y.shape[0], _ptr(x_out), _stream(stream)),
           "clearmoe_layer_norm")


def clearmoe_get_routing(layer: int, idx=None, counts=None, offsets=None, perm=None,
                         stream=None) -> None:
    _check(lib().clearmoe_get_routing(layer, _ptr(idx), _ptr(counts), _ptr(offsets), _ptr(perm),
                                      _stream(stream)), "clearmoe_get_routing")


def clearmoe_layer_status(layer: int) -> int:
    return lib().clearmoe_layer_status(layer)


def clearmoe_debug_set_wait(layer: int, wait_limit_ns: int, phantom_arrivals: int) -> None:
    _check(lib().clearmoe_debug_set_wait(layer, wait_limit_ns, phantom_arrivals),
           "clearmoe_debug_set_wait")


def clearmoe_set_profile_events(layer: int, events) -> None:
    """events: torch.cuda.Event(enable_timing=True) objects (or none to stop recording). torch
    creates an event's CUDA handle on its first record, so each is recorded once here first; the
    library then re-records it on the forward's stream."""
    for e in events:
        if not e.cuda_event:
            e.record()
    handles = [e.cuda_event for e in events]
    arr = (ctypes.c_void_p * max(1, len(handles)))(*handles)
    _check(lib().clearmoe_set_profile_events(layer, arr, len(handles)),
           "clearmoe_set_profile_events")


def clearmoe_route_noalloc(x, Wg, bg, idx, counts, offsets, perm, status=None,
                           stream=None) -> None:
    """Routing without a handle or any device allocation (see include/clearmoe.h): the outputs
    idx [T], counts [E], offsets [E + 1], perm [T] (int32) and the optional status word are
    caller-owned CUDA tensors."""
    import torch
    dtype = BF16 if x.dtype == torch.bfloat16 else F32
    r = _router(Wg, bg)
    _check(lib().clearmoe_route_noalloc(_ptr(x), x.shape[0], x.shape[1], dtype, ctypes.byref(r),
                                        Wg.shape[0], _ptr(idx), _ptr(counts), _ptr(offsets),
                                        _ptr(perm), _ptr(status), _stream(stream)),
           "clearmoe_route_noalloc")
