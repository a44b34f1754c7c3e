"""Python side of the seeded input generator (see gen.c for the definition).

`build()` compiles gen.c with the host gcc into synth/_lib/libsynth.so.
`np_stream_at` / `np_normal` are a plain NumPy restatement of the same
generator, used by the CPU tests to pin the compiled one bit for bit.
"""

import ctypes
import math
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIBDIR = os.path.join(_HERE, "_lib")
_LIB = os.path.join(_LIBDIR, "libsynth.so")
_lib = None

GAMMA = 0x9E3779B97F4A7C15
M64 = (1 << 64) - 1


def build(force=False):
    """Compile gen.c for this host (x86_64 or aarch64), OpenMP enabled."""
    src = os.path.join(_HERE, "gen.c")
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(src):
        return _LIB
    os.makedirs(_LIBDIR, exist_ok=True)
    tmp = _LIB + ".tmp%d" % os.getpid()
    subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared",
                           "-ffp-contract=off", "-o", tmp, src])
    os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB)
        u64, i64, f32, u32 = ctypes.c_uint64, ctypes.c_int64, ctypes.c_float, ctypes.c_uint32
        vp = ctypes.c_void_p
        L.synth_stream_at.argtypes = [u64, u64]
        L.synth_stream_at.restype = u64
        for fn in ("synth_normal_bf16", "synth_normal_f32", "synth_normal_bf16_f64",
                   "synth_normal_f32_f64"):
            getattr(L, fn).argtypes = [u64, u64, i64, f32, vp]
            getattr(L, fn).restype = None
        L.synth_uniform_int.argtypes = [u64, u64, i64, u32, vp]
        L.synth_uniform_int.restype = None
        _lib = L
    return _lib


def mix64(z):
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & M64
    return z ^ (z >> 31)


def stream_at(key, i):
    """i-th output of the SplitMix64 stream keyed by `key` (pure Python)."""
    return mix64((key + (i + 1) * GAMMA) & M64)


def tensor_key(seed, kind, layer=0):
    """Stream key of one tensor: seed -> kind -> layer, each a SplitMix64 step."""
    return stream_at(stream_at(seed & M64, kind), layer)


def ih4_mult(sigma):
    """fp32 multiplier giving std `sigma` to a centred Irwin-Hall(4) 16-bit sum."""
    return float(np.float32(sigma * math.sqrt(3.0) / 65536.0))


_NP_DTYPE = {"bf16": np.uint16, "f32": np.float32, "bf16_f64": np.float64,
             "f32_f64": np.float64}


def normal(key, n, sigma, out_dtype, offset=0, out=None):
    """n approximately normal values of std sigma from stream `key`.

    out_dtype: "bf16" (uint16 bit patterns), "f32", "bf16_f64" (the bf16
    values widened to float64) or "f32_f64".  `out` may be a preallocated
    contiguous array of n elements of the matching dtype.
    """
    L = lib()
    mult = ih4_mult(sigma)
    fn = {"bf16": L.synth_normal_bf16, "f32": L.synth_normal_f32,
          "bf16_f64": L.synth_normal_bf16_f64, "f32_f64": L.synth_normal_f32_f64}[out_dtype]
    if out is None:
        out = np.empty(n, _NP_DTYPE[out_dtype])
    assert out.dtype == _NP_DTYPE[out_dtype] and out.size == n and out.flags.c_contiguous
    fn(key, offset, n, mult, out.ctypes.data)
    return out


def uniform_int(key, n, bound, offset=0):
    out = np.empty(n, np.int32)
    lib().synth_uniform_int(key, offset, n, bound, out.ctypes.data)
    return out


# ---- NumPy restatement (pins the compiled generator in the CPU tests) ----

def np_stream_at(key, idx):
    idx = np.asarray(idx, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(key) + (idx + np.uint64(1)) * np.uint64(GAMMA)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        return z ^ (z >> np.uint64(31))


def np_normal_f32(key, n, sigma, offset=0):
    r = np_stream_at(key, np.arange(offset, offset + n, dtype=np.uint64))
    m = np.uint64(0xFFFF)
    s = ((r & m).astype(np.int64) + ((r >> np.uint64(16)) & m).astype(np.int64) +
         ((r >> np.uint64(32)) & m).astype(np.int64) + (r >> np.uint64(48)).astype(np.int64)
         - 131070)
    return s.astype(np.float32) * np.float32(ih4_mult(sigma))


def np_f32_to_bf16_bits(x):
    u = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    u = u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))
    return (u >> np.uint64(16)).astype(np.uint16)


def bf16_bits_to_f64(b):
    return (np.asarray(b, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def np_uniform_int(key, n, bound, offset=0):
    r = np_stream_at(key, np.arange(offset, offset + n, dtype=np.uint64))
    with np.errstate(over="ignore"):
        return (((r >> np.uint64(32)) * np.uint64(bound)) >> np.uint64(32)).astype(np.int32)
