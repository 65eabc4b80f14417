"""Python binding of the C ABI in include/dlmz.h (argument marshalling only).

Every computation runs in libdlmz.so (CUDA, sm_103a).  Importing this module
raises ``ImportError`` when the library has not been built (there is no
fallback); build it with ``python -m paper_2608_11249_gb300.build``.

Device pointers are passed as integers (e.g. ``tensor.data_ptr()`` of a
torch CUDA tensor) and streams as integer handles (``torch.cuda.Stream
.cuda_stream``; 0 = legacy default stream).
"""
import ctypes
import os
from ctypes import (POINTER, Structure, byref, c_char_p, c_double, c_float, c_int, c_size_t, c_uint8, c_uint32,
                    c_uint64, c_void_p)

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libdlmz.so")
if not os.path.exists(_LIB_PATH):
    raise ImportError("libdlmz.so is not built (python -m paper_2608_11249_gb300.build)")
lib = ctypes.CDLL(_LIB_PATH)

OK, EINVAL, EBADINPUT, ECORRUPT, EMODEL, ENOMEM, ECUDA, ETIMEOUT, ECAPACITY = 0, -1, -2, -3, -4, -5, -6, -7, -8
FP32, BF16 = 0, 1
TOPK_CONF, ENTROPY, UNIFORM, PROGRESSIVE = 0, 1, 2, 3
CONTEXT_NONE, CONTEXT_CONTIGUOUS, CONTEXT_RANDOM, CONTEXT_ATTENTION = 0, 1, 2, 3
CODER_RANGE, CODER_RANS, CODER_RANKS = 0, 1, 2


class DlmzError(RuntimeError):
    def __init__(self, code, where):
        self.code = code
        super().__init__("%s failed: %s (%d)" % (where, lib.dlmz_strerror(code).decode(), code))


class ModelConfig(Structure):
    _fields_ = [("n_layers", c_uint32), ("d", c_uint32), ("n_heads", c_uint32), ("n_kv_heads", c_uint32),
                ("ffn", c_uint32), ("vocab", c_uint32), ("dtype", c_uint32), ("rope_theta", c_float),
                ("norm_eps", c_float), ("seed", c_uint64)]


class KPolicy(Structure):
    _fields_ = [("kind", c_uint32), ("k", c_uint32), ("block", c_uint32), ("tau_bits", c_float),
                ("k_min", c_uint32), ("k_max", c_uint32), ("growth_q16", c_uint32), ("context", c_uint32),
                ("context_c", c_uint32), ("coder", c_uint32), ("context_seed", c_uint64)]


class Profile(Structure):
    _fields_ = [("launches", c_uint64), ("n", c_uint64 * 8), ("ms", c_double * 8), ("flops", c_double * 8),
                ("bytes", c_double * 8)]


def _sig(name, restype, *args):
    f = getattr(lib, name)
    f.restype = restype
    f.argtypes = list(args)
    return f


_P = c_void_p
_sig("dlmz_strerror", c_char_p, c_int)
_sig("dlmz_model_create", c_int, POINTER(ModelConfig), POINTER(c_void_p))
_sig("dlmz_model_destroy", None, _P)
_sig("dlmz_model_fingerprint", c_uint64, _P)
_sig("dlmz_model_get_config", c_int, _P, POINTER(ModelConfig))
_sig("dlmz_model_set_logits_budget", c_int, _P, c_size_t)
_sig("dlmz_compress", c_int, _P, _P, c_size_t, c_uint32, POINTER(KPolicy), POINTER(POINTER(c_uint8)), POINTER(c_size_t))
_sig("dlmz_compress_ex", c_int, _P, _P, c_size_t, c_uint32, POINTER(KPolicy), c_uint32, POINTER(POINTER(c_uint8)),
     POINTER(c_size_t))
_sig("dlmz_decompress", c_int, _P, _P, c_size_t, POINTER(POINTER(c_uint8)), POINTER(c_size_t))
_sig("dlmz_free", None, _P)
_sig("dlmz_compress_bound", c_size_t, _P, c_size_t, c_uint32)
_sig("dlmz_compress_device", c_int, _P, _P, c_size_t, c_uint32, POINTER(KPolicy), c_uint32, _P, c_size_t,
     POINTER(c_size_t), _P)
_sig("dlmz_decompress_device", c_int, _P, _P, c_size_t, _P, c_size_t, POINTER(c_size_t), _P)
_sig("dlmz_forward_logits", c_int, _P, _P, c_uint32, c_uint32, c_uint32, c_uint32, _P, _P)
_sig("dlmz_context_scores", c_int, _P, _P, c_uint32, c_uint32, _P, _P)
_sig("dlmz_gemm_bf16", c_int, _P, _P, _P, c_uint32, c_uint32, c_uint32, _P)
_sig("dlmz_attention_bf16", c_int, _P, c_uint32, c_uint32, c_uint32, c_uint32, c_uint32, c_uint32, _P, _P)
_sig("dlmz_quantize", c_int, _P, c_uint32, c_uint32, c_uint32, _P, _P, _P, _P, _P, _P)
_sig("dlmz_select_smallest", c_int, _P, c_uint32, c_uint32, c_uint32, _P, _P)
_sig("dlmz_select_smallest_noalloc", c_int, _P, c_uint32, c_uint32, c_uint32, _P, _P)
_sig("dlmz_coder_create", c_int, c_uint32, c_uint32, c_uint32, c_uint32, POINTER(c_void_p))
_sig("dlmz_coder_create_ex", c_int, c_uint32, c_uint32, c_uint32, c_uint32, c_uint32, POINTER(c_void_p))
_sig("dlmz_coder_destroy", None, _P)
_sig("dlmz_coder_reset_encoder", c_int, _P, _P)
_sig("dlmz_coder_load_decoder", c_int, _P, _P, _P, _P, _P)
_sig("dlmz_encode_step", c_int, _P, POINTER(KPolicy), _P, c_uint32, c_uint32, _P, _P, _P, _P)
_sig("dlmz_decode_step", c_int, _P, POINTER(KPolicy), _P, c_uint32, c_uint32, _P, _P, _P)
_sig("dlmz_coder_finish", c_int, _P, _P, _P, _P, _P)
_sig("dlmz_model_encode_step", c_int, _P, _P, POINTER(KPolicy), c_uint32, c_uint32, _P, _P, _P, _P)
_sig("dlmz_model_decode_step", c_int, _P, _P, POINTER(KPolicy), c_uint32, c_uint32, _P, _P, _P)
_sig("dlmz_coder_capacity_units", c_uint32, _P)
_sig("dlmz_check", c_int, _P)
_sig("dlmz_selftest_wait_timeout", c_int, c_uint32, _P)
_sig("dlmz_selftest_cluster_wait", c_int, c_uint32, c_uint32, _P)
_sig("dlmz_profile_begin", c_int)
_sig("dlmz_profile_end", c_int, POINTER(Profile))
_sig("dlmz_launch_count", c_uint64)


def _ok(rc, where):
    if rc != OK:
        raise DlmzError(rc, where)


def strerror(code):
    return lib.dlmz_strerror(code).decode()


def policy(kind=TOPK_CONF, k=1, block=0, tau_bits=0.0, k_min=1, k_max=0, growth_q16=65536,
           context=CONTEXT_NONE, context_c=0, context_seed=0, coder=0):
    return KPolicy(kind, k, block, tau_bits, k_min, k_max, growth_q16, context, context_c, coder, context_seed)


class Model:
    """Owns a dlmz_model (random-init masked DLM on the current CUDA device)."""

    def __init__(self, n_layers, d, n_heads, n_kv_heads, ffn, vocab, dtype=BF16, rope_theta=10000.0,
                 norm_eps=1e-5, seed=0):
        self.cfg = ModelConfig(n_layers, d, n_heads, n_kv_heads, ffn, vocab, dtype, rope_theta, norm_eps, seed)
        h = c_void_p()
        _ok(lib.dlmz_model_create(byref(self.cfg), byref(h)), "dlmz_model_create")
        self.h = h

    def close(self):
        if self.h:
            lib.dlmz_model_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def fingerprint(self):
        return lib.dlmz_model_fingerprint(self.h)

    def set_logits_budget(self, nbytes):
        """Bytes of candidate logits one step holds at once (0: the library default)."""
        _ok(lib.dlmz_model_set_logits_budget(self.h, nbytes), "dlmz_model_set_logits_budget")

    def compress(self, data, chunk_len, pol, batch_chunks=0):
        buf = bytes(data)
        out = POINTER(c_uint8)()
        n = c_size_t()
        rc = lib.dlmz_compress_ex(self.h, buf, len(buf), chunk_len, byref(pol), batch_chunks, byref(out), byref(n))
        _ok(rc, "dlmz_compress")
        try:
            return ctypes.string_at(out, n.value)
        finally:
            lib.dlmz_free(out)

    def decompress(self, blob):
        blob = bytes(blob)
        out = POINTER(c_uint8)()
        n = c_size_t()
        _ok(lib.dlmz_decompress(self.h, blob, len(blob), byref(out), byref(n)), "dlmz_decompress")
        try:
            return ctypes.string_at(out, n.value)
        finally:
            lib.dlmz_free(out)

    def compress_bound(self, in_bytes, chunk_len):
        return lib.dlmz_compress_bound(self.h, in_bytes, chunk_len)

    def compress_device(self, d_in, in_bytes, chunk_len, pol, d_out, out_cap, batch_chunks=0, stream=0):
        n = c_size_t()
        _ok(lib.dlmz_compress_device(self.h, d_in, in_bytes, chunk_len, byref(pol), batch_chunks, d_out, out_cap,
                                     byref(n), stream), "dlmz_compress_device")
        return n.value

    def decompress_device(self, d_in, in_bytes, d_out, out_cap, stream=0):
        n = c_size_t()
        _ok(lib.dlmz_decompress_device(self.h, d_in, in_bytes, d_out, out_cap, byref(n), stream),
            "dlmz_decompress_device")
        return n.value

    def forward_logits(self, d_state, n_chunks, L, row0, rows_per_chunk, d_logits, stream=0):
        _ok(lib.dlmz_forward_logits(self.h, d_state, n_chunks, L, row0, rows_per_chunk, d_logits, stream),
            "dlmz_forward_logits")

    def encode_step(self, coder, pol, row0, rpc, d_symbols, d_state, d_committed=None, stream=0):
        """One denoising step with this model's distributions, coding into ``coder`` (a Coder)."""
        _ok(lib.dlmz_model_encode_step(self.h, coder.h, byref(pol), row0, rpc, d_symbols, d_state, d_committed,
                                       stream), "dlmz_model_encode_step")

    def decode_step(self, coder, pol, row0, rpc, d_state, d_committed=None, stream=0):
        _ok(lib.dlmz_model_decode_step(self.h, coder.h, byref(pol), row0, rpc, d_state, d_committed, stream),
            "dlmz_model_decode_step")

    def context_scores(self, d_symbols, n_chunks, L, d_scores, stream=0):
        _ok(lib.dlmz_context_scores(self.h, d_symbols, n_chunks, L, d_scores, stream), "dlmz_context_scores")


def gemm_bf16(d_A, d_B, d_D, M, N, K, stream=0):
    _ok(lib.dlmz_gemm_bf16(d_A, d_B, d_D, M, N, K, stream), "dlmz_gemm_bf16")


def attention_bf16(d_qkv, ld, n_chunks, L, n_heads, n_kv_heads, head_dim, d_out, stream=0):
    _ok(lib.dlmz_attention_bf16(d_qkv, ld, n_chunks, L, n_heads, n_kv_heads, head_dim, d_out, stream),
        "dlmz_attention_bf16")


def quantize(d_logits, rows, V, P, d_cdf, d_W, d_A, d_Hq, d_top, stream=0):
    _ok(lib.dlmz_quantize(d_logits, rows, V, P, d_cdf, d_W, d_A, d_Hq, d_top, stream), "dlmz_quantize")


def select_smallest(d_keys, groups, group_size, k, d_out, stream=0):
    _ok(lib.dlmz_select_smallest(d_keys, groups, group_size, k, d_out, stream), "dlmz_select_smallest")


def select_smallest_noalloc(d_keys, groups, group_size, k, d_out, stream=0):
    """dlmz_select_smallest without any device allocation (static scratch, <= 65536 groups)."""
    _ok(lib.dlmz_select_smallest_noalloc(d_keys, groups, group_size, k, d_out, stream),
        "dlmz_select_smallest_noalloc")


def profile_begin():
    _ok(lib.dlmz_profile_begin(), "dlmz_profile_begin")


def profile_end(prof):
    _ok(lib.dlmz_profile_end(byref(prof)), "dlmz_profile_end")


def launch_count():
    """Kernels launched by the library so far (dlmz_launch_count)."""
    return int(lib.dlmz_launch_count())


def check(stream=0):
    _ok(lib.dlmz_check(stream), "dlmz_check")


def selftest_wait_timeout(limit_us, stream=0):
    """Return code of dlmz_selftest_wait_timeout (DLMZ_ETIMEOUT when the bounded wait gave up)."""
    return lib.dlmz_selftest_wait_timeout(limit_us, stream)


def selftest_cluster_wait(limit_us, peer_arrives, stream=0):
    """Return code of dlmz_selftest_cluster_wait (OK when the peer CTA arrived, ETIMEOUT when not)."""
    return lib.dlmz_selftest_cluster_wait(limit_us, peer_arrives, stream)


class Coder:
    """Owns a dlmz_coder: one coder stream (range coder or rANS) per window of a batch."""

    def __init__(self, n_chunks, L, V, P, coder=CODER_RANGE):
        h = c_void_p()
        _ok(lib.dlmz_coder_create_ex(n_chunks, L, V, P, coder, byref(h)), "dlmz_coder_create_ex")
        self.h = h

    def close(self):
        if self.h:
            lib.dlmz_coder_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def capacity_units(self):
        return lib.dlmz_coder_capacity_units(self.h)

    def reset_encoder(self, stream=0):
        _ok(lib.dlmz_coder_reset_encoder(self.h, stream), "dlmz_coder_reset_encoder")

    def load_decoder(self, d_bytes, d_offsets, d_bits, stream=0):
        _ok(lib.dlmz_coder_load_decoder(self.h, d_bytes, d_offsets, d_bits, stream), "dlmz_coder_load_decoder")

    def encode_step(self, pol, d_logits, row0, rpc, d_symbols, d_state, d_committed=None, stream=0):
        _ok(lib.dlmz_encode_step(self.h, byref(pol), d_logits, row0, rpc, d_symbols, d_state, d_committed, stream),
            "dlmz_encode_step")

    def decode_step(self, pol, d_logits, row0, rpc, d_state, d_committed=None, stream=0):
        _ok(lib.dlmz_decode_step(self.h, byref(pol), d_logits, row0, rpc, d_state, d_committed, stream),
            "dlmz_decode_step")

    def finish(self, d_bits, d_bytes=None, d_offsets=None, stream=0):
        _ok(lib.dlmz_coder_finish(self.h, d_bits, d_bytes, d_offsets, stream), "dlmz_coder_finish")
