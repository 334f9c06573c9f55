"""ctypes loader of the plain-C float64 oracle (oracle/clearmoe_ref.c). TEST INFRASTRUCTURE ONLY.

The shared library is compiled with the host's gcc on first use (or by the repository's build
step) into oracle/libclearmoe_ref.so, with floating-point contraction off so that x86 and Arm
hosts give the same bits. Every wrapper takes and returns numpy arrays (float64, row-major); the
arithmetic is all in the C file.
"""
from __future__ import annotations

import ctypes
import pathlib
import shutil
import subprocess

import numpy as np

HERE = pathlib.Path(__file__).resolve().parent
SRC = HERE / "clearmoe_ref.c"
LIB = HERE / "libclearmoe_ref.so"
CFLAGS = ["-std=c99", "-O2", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math"]

_lib = None
_D = ctypes.POINTER(ctypes.c_double)
_I = ctypes.POINTER(ctypes.c_int32)
_SIGS = {
    "cmref_round_bf16": (ctypes.c_double, [ctypes.c_double]),
    "cmref_gelu": (ctypes.c_double, [ctypes.c_double]),
    "cmref_router_logits": (None, [_D, ctypes.c_int64, ctypes.c_int, _D, _D, ctypes.c_int, _D]),
    "cmref_mlp_router_logits": (None, [_D, ctypes.c_int64, ctypes.c_int, _D, _D, ctypes.c_int, _D, _D,
                                       ctypes.c_int, ctypes.c_int, _D]),
    "cmref_argmax": (None, [_D, ctypes.c_int64, ctypes.c_int, ctypes.c_int64, _I]),
    "cmref_sort_by_group": (ctypes.c_int, [_I, ctypes.c_int64, ctypes.c_int, _I, _I, _I]),
    "cmref_fc1_gelu": (None, [_D, ctypes.c_int64, ctypes.c_int, ctypes.c_int, _D, _D, ctypes.c_int, _D]),
    "cmref_shared_weight": (None, [_D, _D, _D, ctypes.c_int, ctypes.c_int, ctypes.c_int, _D]),
    "cmref_experts_forward": (ctypes.c_int, [_D, ctypes.c_int64, ctypes.c_int, ctypes.c_int, _D, _D,
                                             ctypes.c_int, _I, _D, _D, _D]),
    "cmref_ffn_forward": (ctypes.c_int, [_D, ctypes.c_int64, ctypes.c_int, ctypes.c_int, _D, _D, _D, _D, _D,
                                         ctypes.c_int, _D, ctypes.c_int, _I, _D, _D, ctypes.c_int, _D]),
    "cmref_dense_ffn": (ctypes.c_int, [_D, ctypes.c_int64, ctypes.c_int, ctypes.c_int, _D, _D, _D, _D,
                                       ctypes.c_int, _D]),
    "cmref_layer_norm": (None, [_D, ctypes.c_int64, ctypes.c_int, ctypes.c_double, _D]),
    "cmref_fold_basis": (None, [_D, _D, _D, _D, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, _D]),
    "cmref_ffn_forward_scaled": (ctypes.c_int, [_D, ctypes.c_int64, ctypes.c_int, ctypes.c_int, _D, _D, _D, _D,
                                                _D, ctypes.c_int, _D, _D, ctypes.c_int, _I, ctypes.c_int, _D]),
}


def compile_ref(force: bool = False) -> pathlib.Path:
    """gcc -> oracle/libclearmoe_ref.so (skipped while the library is newer than its source)."""
    if LIB.exists() and not force and LIB.stat().st_mtime >= SRC.stat().st_mtime:
        return LIB
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        raise RuntimeError("no C compiler found for the C oracle")
    tmp = LIB.with_suffix(".so.tmp")
    r = subprocess.run([cc, *CFLAGS, "-o", str(tmp), str(SRC), "-lm"], capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"gcc failed on {SRC.name}:\n{r.stdout}\n{r.stderr}")
    tmp.replace(LIB)
    return LIB


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        h = ctypes.CDLL(str(compile_ref()))
        for name, (res, args) in _SIGS.items():
            fn = getattr(h, name)
            fn.restype = res
            fn.argtypes = args
        _lib = h
    return _lib


def _d(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def _p(a):
    return None if a is None else a.ctypes.data_as(_D)


def _pi(a):
    return a.ctypes.data_as(_I)


def round_bf16(v) -> np.ndarray:
    f = lib().cmref_round_bf16
    return np.vectorize(f, otypes=[np.float64])(_d(v))


def gelu(u) -> np.ndarray:
    f = lib().cmref_gelu
    return np.vectorize(f, otypes=[np.float64])(_d(u))


def router_logits(x, Wg, bg) -> np.ndarray:
    x, Wg, bg = _d(x), _d(Wg), _d(bg)
    T, d = x.shape
    out = np.empty((T, Wg.shape[0]))
    lib().cmref_router_logits(_p(x), T, d, _p(Wg), _p(bg), Wg.shape[0], _p(out))
    return out


def mlp_router_logits(x, W_in, b_in, W_out, b_out, act: str = "relu") -> np.ndarray:
    x, W_in, b_in, W_out, b_out = (_d(v) for v in (x, W_in, b_in, W_out, b_out))
    T, d = x.shape
    out = np.empty((T, W_out.shape[0]))
    lib().cmref_mlp_router_logits(_p(x), T, d, _p(W_in), _p(b_in), W_in.shape[0], _p(W_out), _p(b_out),
                                  W_out.shape[0], {"relu": 0, "gelu": 1}[act], _p(out))
    return out


def argmax(logits, cls_stride: int = 0) -> np.ndarray:
    lg = _d(logits)
    a = np.empty(lg.shape[0], np.int32)
    lib().cmref_argmax(_p(lg), lg.shape[0], lg.shape[1], int(cls_stride), _pi(a))
    return a.astype(np.int64)


def route(x, Wg, bg, cls_stride: int = 0) -> dict:
    """Expert (or class group) per token on float64 logits, then the stable sort by group."""
    a = argmax(router_logits(x, Wg, bg), cls_stride)
    return sort_by_group(a, np.asarray(Wg).shape[0] + (1 if cls_stride else 0))


def sort_by_group(a, G: int) -> dict:
    a32 = np.ascontiguousarray(a, dtype=np.int32)
    counts, offsets, perm = np.empty(G, np.int32), np.empty(G + 1, np.int32), np.empty(a32.size, np.int32)
    if lib().cmref_sort_by_group(_pi(a32), a32.size, G, _pi(counts), _pi(offsets), _pi(perm)):
        raise ValueError("group index outside [0, G)")
    return dict(a=a32.astype(np.int64), counts=counts.astype(np.int64), offsets=offsets.astype(np.int64),
                perm=perm.astype(np.int64))


def fc1_gelu(x, W1, b1, z_bf16: bool = False) -> np.ndarray:
    x, W1, b1 = _d(x), _d(W1), _d(b1)
    T, d = x.shape
    z = np.empty((T, W1.shape[0]))
    lib().cmref_fc1_gelu(_p(x), T, d, W1.shape[0], _p(W1), _p(b1), int(z_bf16), _p(z))
    return z


def shared_weight(U, S, Vh) -> np.ndarray:
    U, S, Vh = _d(U), _d(S), _d(Vh)
    out = np.empty((U.shape[0], Vh.shape[1]))
    lib().cmref_shared_weight(_p(U), _p(S), _p(Vh), U.shape[0], U.shape[1], Vh.shape[1], _p(out))
    return out


def ffn_forward(x, W1, b1, U, S, Vh, residuals, a, W2=None, b2=None, z_bf16: bool = False) -> np.ndarray:
    """Eq. 2 / Algorithm 3 for the given groups a (a_t = E: class token, dense path W2)."""
    x, W1, b1, U, S, Vh, res = (_d(v) for v in (x, W1, b1, U, S, Vh, residuals))
    W2 = None if W2 is None else _d(W2)
    b2 = None if b2 is None else _d(b2)
    a32 = np.ascontiguousarray(a, dtype=np.int32)
    T, d = x.shape
    y = np.empty((T, d))
    rc = lib().cmref_ffn_forward(_p(x), T, d, W1.shape[0], _p(W1), _p(b1), _p(U), _p(S), _p(Vh), S.shape[0],
                                 _p(res), res.shape[0], _pi(a32), _p(W2), _p(b2), int(z_bf16), _p(y))
    if rc:
        raise ValueError("bad group index or allocation failure")
    return y


def dense_ffn(x, W1, b1, W2, b2=None, z_bf16: bool = False) -> np.ndarray:
    x, W1, b1, W2 = (_d(v) for v in (x, W1, b1, W2))
    b2 = None if b2 is None else _d(b2)
    T, d = x.shape
    y = np.empty((T, d))
    if lib().cmref_dense_ffn(_p(x), T, d, W1.shape[0], _p(W1), _p(b1), _p(W2), _p(b2), int(z_bf16), _p(y)):
        raise MemoryError("allocation failure")
    return y


def layer_norm(y, eps: float = 1e-6) -> np.ndarray:
    y = _d(y)
    T, d = y.shape
    out = np.empty_like(y)
    lib().cmref_layer_norm(_p(y), T, d, float(eps), _p(out))
    return out


def fold_basis(U, S, Vh, residuals) -> np.ndarray:
    """W_comb[e] = W_shared + W_e^res for every expert."""
    U, S, Vh, res = (_d(v) for v in (U, S, Vh, residuals))
    E, d, H = res.shape
    out = np.empty((E, d, H))
    lib().cmref_fold_basis(_p(U), _p(S), _p(Vh), _p(res), E, d, S.shape[0], H, _p(out))
    return out


def ffn_forward_scaled(x, W1, b1, U, S, Vh, R, s, a, z_bf16: bool = False) -> np.ndarray:
    """y_t = W_shared z_t + s_{a_t} R z_t (Algorithm 2's residuals W_e^res = s_e R)."""
    x, W1, b1, U, S, Vh, R, s = (_d(v) for v in (x, W1, b1, U, S, Vh, R, s))
    a32 = np.ascontiguousarray(a, dtype=np.int32)
    T, d = x.shape
    y = np.empty((T, d))
    if lib().cmref_ffn_forward_scaled(_p(x), T, d, W1.shape[0], _p(W1), _p(b1), _p(U), _p(S), _p(Vh), S.shape[0],
                                      _p(R), _p(s), s.shape[0], _pi(a32), int(z_bf16), _p(y)):
        raise ValueError("bad expert index or allocation failure")
    return y
