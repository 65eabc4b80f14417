"""Counter-based random initialisation of the model weights (oracle side).

The paper evaluates a trained LLaDA-8B (Sec. 4, "Implementation Details");
trained weights are not available, so every model here is randomly
initialised with N(0, 0.02) entries.  Norm gains are 1.

The generator is defined by published algorithms so that the CUDA library
can regenerate the same values independently:

* SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number
  generators", OOPSLA 2014): the n-th output (n = 0, 1, ...) of a stream
  with state ``s`` is ``mix(s + (n + 1) * GAMMA)``.
* Tensor ``tid`` of a model with seed ``seed`` uses the stream whose state is
  the ``tid``-th output of the stream with state ``seed``.
* Basic Box-Muller transform (Box & Muller 1958): element pair ``(2j, 2j+1)``
  takes outputs ``u0 = out[2j]``, ``u1 = out[2j+1]``;
  ``a = ((u0 >> 11) + 1) * 2^-53`` in (0, 1], ``b = (u1 >> 11) * 2^-53``;
  ``r = sqrt(-2 ln a)``, ``z[2j] = r cos(2 pi b)``, ``z[2j+1] = r sin(2 pi b)``.
* weight = ``0.02 * z`` in float64, then rounded (RNE) to the model's storage
  dtype (float32 or bfloat16).

Element ``n`` of a tensor is its row-major index in the logical shape given
in ``model.tensor_shapes``.

Parity: pinned by tests of the SplitMix64 reference outputs, of the sample
moments, and of the Box-Muller identity z0^2 + z1^2 = -2 ln a.
"""
import math

import numpy as np

GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
STD = 0.02


def mix64(z):
    """SplitMix64 output function on a uint64 array (wrapping arithmetic)."""
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def stream_outputs(state, n0, count):
    """Outputs n0 .. n0+count-1 of the SplitMix64 stream with ``state``."""
    idx = np.arange(n0 + 1, n0 + count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return mix64(np.uint64(state) + idx * GAMMA)


def tensor_state(seed, tid):
    """State of the stream of tensor ``tid``: output ``tid`` of the seed stream."""
    return int(stream_outputs(np.uint64(seed), tid, 1)[0])


def normal_draws(seed, tid, count):
    """``count`` standard-normal draws (float64) for tensor ``tid``."""
    npairs = (count + 1) // 2
    u = stream_outputs(tensor_state(seed, tid), 0, 2 * npairs)
    u0 = u[0::2]
    u1 = u[1::2]
    a = ((u0 >> np.uint64(11)) + np.uint64(1)).astype(np.float64) * 2.0 ** -53
    b = (u1 >> np.uint64(11)).astype(np.float64) * 2.0 ** -53
    r = np.sqrt(-2.0 * np.log(a))
    t = math.tau * b
    z = np.empty(2 * npairs, dtype=np.float64)
    z[0::2] = r * np.cos(t)
    z[1::2] = r * np.sin(t)
    return z[:count]


def round_bf16(x):
    """Round float64 values to the nearest bfloat16 (ties to even).

    bfloat16 keeps 8 significant bits and float32's exponent range; the
    float64 significand is rounded to 8 bits directly (no intermediate
    float32 rounding).  Valid for |x| in the bfloat16 normal range and 0.
    """
    x = np.ascontiguousarray(x, dtype=np.float64)
    b = x.view(np.uint64)
    drop = np.uint64(45)  # 52 - 7 explicit mantissa bits dropped
    lsb = (b >> drop) & np.uint64(1)
    half = np.uint64((1 << 44) - 1)
    with np.errstate(over="ignore"):
        r = (b + half + lsb) & ~np.uint64((1 << 45) - 1)
    return r.view(np.float64)


def round_f32(x):
    """Round float64 values to the nearest float32 (ties to even)."""
    return np.asarray(x, dtype=np.float64).astype(np.float32).astype(np.float64)


def storage_round(x, dtype):
    """Round to the storage dtype of the model ('f32' or 'bf16')."""
    if dtype == "bf16":
        return round_bf16(x)
    if dtype == "f32":
        return round_f32(x)
    raise ValueError(dtype)


def init_tensor(seed, tid, shape, dtype):
    """Weights of tensor ``tid`` with logical row-major ``shape``."""
    n = int(np.prod(shape))
    z = normal_draws(seed, tid, n) * STD
    return storage_round(z, dtype).reshape(shape)


# ---- the same draws in plain C (oracle/csrc/normal_draws.c), for full-size models ----------
_NATIVE = None


def _native():
    """ctypes handle of liboracle.so (built by oracle/build.py), or None when it is not built."""
    global _NATIVE
    if _NATIVE is None:
        import ctypes
        import os
        path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "liboracle.so")
        if not os.path.exists(path):
            return None
        lib = ctypes.CDLL(path)
        lib.oracle_normal_range.restype = None
        lib.oracle_normal_range.argtypes = [ctypes.c_uint64, ctypes.c_int64, ctypes.c_int64, ctypes.c_double,
                                            ctypes.c_int, ctypes.c_void_p]
        _NATIVE = lib
    return _NATIVE


_MODES = {None: 0, "f32": 1, "bf16": 2}


def normal_draws_c(seed, tid, count, n0=0, threads=None, scale=1.0, dtype=None):
    """Draws n0 .. n0+count-1 of tensor ``tid`` (as ``normal_draws``) times ``scale``,
    rounded to ``dtype`` (None: no rounding), computed by the C restatement on
    ``threads`` host threads (ctypes releases the interpreter lock)."""
    import concurrent.futures as cf
    import os
    lib = _native()
    if lib is None:
        raise RuntimeError("liboracle.so is not built (python oracle/build.py)")
    out = np.empty(count, dtype=np.float64)
    st = tensor_state(seed, tid)
    if threads is None:
        threads = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
    step = max(1 << 20, -(-count // max(1, threads)))
    step += step & 1
    base = out.ctypes.data

    def run(a):
        b = min(count, a + step)
        lib.oracle_normal_range(st, n0 + a, b - a, scale, _MODES[dtype], base + 8 * a)

    with cf.ThreadPoolExecutor(max_workers=max(1, threads)) as ex:
        list(ex.map(run, range(0, count, step)))
    return out


def init_tensor_c(seed, tid, shape, dtype):
    """``init_tensor`` with the draws from the C restatement (same values up to the last
    bits of the float64 log / cos / sin, so equal after rounding to bf16 except with
    probability ~2^-44 per element)."""
    n = int(np.prod(shape))
    return normal_draws_c(seed, tid, n, scale=STD, dtype=dtype).reshape(shape)
