"""ctypes binding of libqk (include/qk.h): the same entry points, argument marshalling only.

Device buffers may be passed as torch CUDA tensors (their data_ptr() is used)
or as raw integer addresses; ``None`` passes NULL.  ``stream`` defaults to
torch's current CUDA stream.  A non-zero status raises QKError carrying
qk_last_error().
"""
from __future__ import annotations

import ctypes
import os

PKG = os.path.dirname(os.path.abspath(__file__))
_LIB_FILE = os.path.join(PKG, "libqk.so")

QK_OK, QK_EINVAL, QK_ESHAPE, QK_EDTYPE, QK_ECUDA, QK_ETIMEOUT, QK_EDEVICE, QK_ENOSPACE = (
    0, -1, -2, -3, -4, -5, -6, -7)
QK_DTYPE_BF16, QK_DTYPE_F32 = 0, 1
QK_STATUS_BAD_TOKEN, QK_STATUS_BAD_POS, QK_STATUS_TIMEOUT, QK_STATUS_BAD_PAGE = 1, 2, 4, 8
QK_CALL_DECODE, QK_CALL_PREFILL, QK_CALL_SCORE, QK_CALL_ROLLOUT, QK_CALL_BACKWARD = 0, 1, 2, 3, 4
QK_PROF_QKV, QK_PROF_O, QK_PROF_GATE_UP, QK_PROF_DOWN, QK_PROF_ATTN, QK_PROF_LM_HEAD = range(6)
QK_EPI_STORE, QK_EPI_STORE_F32, QK_EPI_RESID_F32, QK_EPI_SWIGLU = 0, 1, 2, 3
QK_STATIC_SCRATCH_BYTES = 8 << 20

__all__ = [
    "QK_OK", "QK_EINVAL", "QK_ESHAPE", "QK_EDTYPE", "QK_ECUDA", "QK_ETIMEOUT", "QK_EDEVICE",
    "QK_ENOSPACE", "QK_DTYPE_BF16", "QK_DTYPE_F32", "QK_STATUS_BAD_TOKEN", "QK_STATUS_BAD_POS",
    "QK_STATUS_TIMEOUT", "QK_CALL_DECODE", "QK_CALL_PREFILL", "QK_CALL_SCORE", "QK_CALL_ROLLOUT",
    "qk_config", "qk_config_preset", "qk_weight_count", "qk_model_packed_bytes", "qk_model_load",
    "qk_model_free", "qk_kv_bytes", "qk_workspace_bytes", "qk_prefill", "qk_decode_step",
    "qk_decode_layer", "qk_score_logprobs", "qk_rollout_teacher_forced", "qk_check_status",
    "qk_last_error", "QKError", "lib_path", "exported_symbols", "qk_profile_begin",
    "qk_profile_end", "qk_launch_count", "qk_op_linear", "QK_PROF_QKV", "QK_PROF_O",
    "QK_PROF_GATE_UP", "QK_PROF_DOWN", "QK_PROF_ATTN", "QK_PROF_LM_HEAD", "QK_EPI_STORE",
    "QK_EPI_STORE_F32", "QK_EPI_RESID_F32", "QK_EPI_SWIGLU", "qk_op_linear_swiglu_static",
    "QK_STATIC_SCRATCH_BYTES", "qk_grpo_workspace_bytes", "qk_grpo_token_loss", "qk_score_grpo",
    "qk_rollout_sampled", "qk_prefill_rows", "qk_debug_expire_next_wait", "QK_CALL_BACKWARD",
    "qk_grpo_coef", "qk_backward_logprob", "QK_STATUS_BAD_PAGE", "qk_kv_pages", "qk_kv_pages_bytes",
    "qk_decode_step_paged", "qk_prefill_rows_paged", "qk_rollout_teacher_forced_paged",
    "qk_rollout_sampled_paged",
]


class QKError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"libqk error {code}: {msg}")
        self.code = code


class qk_config(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("hidden", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("intermediate", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("max_positions", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("rms_eps", ctypes.c_double), ("rope_theta", ctypes.c_double)]

    def __repr__(self):
        return "qk_config(" + ", ".join(f"{n}={getattr(self, n)}" for n, _ in self._fields_) + ")"


class qk_kv_pages(ctypes.Structure):
    """Paged cache layout: table (device int32 [B, per_row] page ids), per_row,
    n_pages, page_size (a multiple of 128)."""
    _fields_ = [("table", ctypes.c_void_p), ("per_row", ctypes.c_int32),
                ("n_pages", ctypes.c_int32), ("page_size", ctypes.c_int32)]


def lib_path() -> str:
    return _LIB_FILE


_P, _I, _SZ, _F = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_float
_SIGS = {
    "qk_config_preset": ([ctypes.c_char_p, ctypes.POINTER(qk_config)], _I),
    "qk_weight_count": ([ctypes.POINTER(qk_config), ctypes.POINTER(_I)], _I),
    "qk_model_packed_bytes": ([ctypes.POINTER(qk_config), ctypes.POINTER(_SZ)], _I),
    "qk_model_load": ([ctypes.POINTER(qk_config), ctypes.POINTER(_P), _I, _P, _SZ, _P,
                       ctypes.POINTER(_P)], _I),
    "qk_model_free": ([_P], None),
    "qk_kv_bytes": ([_P, _I, _I, ctypes.POINTER(_SZ)], _I),
    "qk_workspace_bytes": ([_P, _I, _I, _I, _I, ctypes.POINTER(_SZ)], _I),
    "qk_prefill": ([_P, _P, _I, _I, _P, _I, _I, _I, _P, _P, _P, _P, _P, _SZ, _P], _I),
    "qk_decode_step": ([_P, _P, _I, _I, _P, _P, _I, _P, _P, _P, _P, _P, _SZ, _P], _I),
    "qk_decode_layer": ([_P, _I, _P, _I, _I, _P, _P, _I, _P, _SZ, _P], _I),
    "qk_score_logprobs": ([_P, _P, _I, _I, _P, _P, _P, _SZ, _P], _I),
    "qk_rollout_teacher_forced": ([_P, _P, _I, _I, _P, _I, _I, _I, _P, _P, _P, _SZ, _P], _I),
    "qk_check_status": ([_P, _P, ctypes.POINTER(ctypes.c_uint32)], _I),
    "qk_last_error": ([], ctypes.c_char_p),
    "qk_profile_begin": ([_P, _I, _I], _I),
    "qk_profile_end": ([_P, ctypes.POINTER(ctypes.c_float), ctypes.POINTER(_I)], _I),
    "qk_launch_count": ([], ctypes.c_uint64),
    "qk_op_linear": ([_P, _P, _I, _P, _P, _I, _I, _I, _I, _I, _P, _SZ, _P], _I),
    "qk_op_linear_swiglu_static": ([_P, _P, _I, _P, _P, _I, _I, _I, _I, _P], _I),
    "qk_grpo_workspace_bytes": ([_I, ctypes.POINTER(_SZ)], _I),
    "qk_grpo_token_loss": ([_P, _P, _P, _I, _I, _I, _P, _I, _P, _F, _F, _F, _P, _P, _P, _SZ, _P], _I),
    "qk_score_grpo": ([_P, _P, _I, _I, _P, _P, _P, _I, _P, _F, _F, _F, _P, _P, _P, _P, _SZ, _P], _I),
    "qk_rollout_sampled": ([_P, _P, _I, _I, _P, _I, _I, _I, _F, ctypes.c_uint64, _P, _P, _P, _SZ, _P],
                           _I),
    "qk_prefill_rows": ([_P, _P, _I, _I, _P, _I, _I, _P, _P, _P, _P, _SZ, _P], _I),
    "qk_debug_expire_next_wait": ([_P, ctypes.c_longlong], _I),
    "qk_grpo_coef": ([_P, _P, _P, _I, _I, _I, _P, _I, _P, _F, _F, _F, _P, _P, _P, _P, _SZ, _P], _I),
    "qk_backward_logprob": ([_P, _P, _I, _I, _P, ctypes.POINTER(_P), _I, _I, _P, _P, _SZ, _P], _I),
    "qk_kv_pages_bytes": ([_P, _I, _I, ctypes.POINTER(_SZ)], _I),
    "qk_rollout_teacher_forced_paged": ([_P, _P, ctypes.POINTER(qk_kv_pages), _P, _I, _I, _I, _P, _P, _P,
                                         _SZ, _P], _I),
    "qk_rollout_sampled_paged": ([_P, _P, ctypes.POINTER(qk_kv_pages), _P, _I, _I, _I, _F, ctypes.c_uint64,
                                  _P, _P, _P, _SZ, _P], _I),
    "qk_decode_step_paged": ([_P, _P, ctypes.POINTER(qk_kv_pages), _P, _P, _I, _P, _P, _P, _P, _P, _SZ,
                              _P], _I),
    "qk_prefill_rows_paged": ([_P, _P, ctypes.POINTER(qk_kv_pages), _P, _I, _I, _P, _P, _P, _P, _SZ, _P],
                              _I),
}

_lib = None


def _load():
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_FILE):
            raise ImportError(f"libqk.so is not built ({_LIB_FILE}); run "
                              "paper_2609_12471_gb300.build.build() or __graft_entry__.build()")
        lib = ctypes.CDLL(_LIB_FILE)
        for name, (args, res) in _SIGS.items():
            f = getattr(lib, name)
            f.argtypes = args
            f.restype = res
        _lib = lib
    return _lib


def exported_symbols():
    """Names of the ABI entry points this binding resolves (all must exist in libqk.so)."""
    lib = _load()
    return [n for n in _SIGS if hasattr(lib, n)]


def qk_last_error() -> str:
    return _load().qk_last_error().decode()


def _check(rc: int):
    if rc != QK_OK:
        raise QKError(rc, qk_last_error())


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    raise TypeError(f"cannot pass {type(x)} as a pointer")


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _nbytes(t, given):
    if given is not None:
        return given
    return t.numel() * t.element_size()


def qk_config_preset(name: str) -> qk_config:
    c = qk_config()
    _check(_load().qk_config_preset(name.encode(), ctypes.byref(c)))
    return c


def qk_weight_count(cfg: qk_config) -> int:
    n = _I()
    _check(_load().qk_weight_count(ctypes.byref(cfg), ctypes.byref(n)))
    return n.value


def qk_model_packed_bytes(cfg: qk_config) -> int:
    n = _SZ()
    _check(_load().qk_model_packed_bytes(ctypes.byref(cfg), ctypes.byref(n)))
    return n.value


def qk_model_load(cfg: qk_config, tensors, packed, packed_bytes=None, stream=None):
    arr = (_P * len(tensors))(*[_ptr(t) for t in tensors])
    out = _P()
    _check(_load().qk_model_load(ctypes.byref(cfg), arr, len(tensors), _ptr(packed),
                                 _nbytes(packed, packed_bytes), _stream(stream), ctypes.byref(out)))
    return out.value


def qk_model_free(m):
    _load().qk_model_free(m)


def qk_kv_bytes(m, max_batch: int, max_seq: int) -> int:
    n = _SZ()
    _check(_load().qk_kv_bytes(m, max_batch, max_seq, ctypes.byref(n)))
    return n.value


def qk_workspace_bytes(m, kind: int, B: int, T: int, max_seq: int) -> int:
    n = _SZ()
    _check(_load().qk_workspace_bytes(m, kind, B, T, max_seq, ctypes.byref(n)))
    return n.value


def qk_prefill(m, kv, max_batch, max_seq, tokens, B, T, start_pos=0, last_logits=None,
               targets=None, logprobs=None, argmax=None, workspace=None, ws_bytes=None,
               stream=None):
    _check(_load().qk_prefill(m, _ptr(kv), max_batch, max_seq, _ptr(tokens), B, T, start_pos,
                              _ptr(last_logits), _ptr(targets), _ptr(logprobs), _ptr(argmax),
                              _ptr(workspace), _nbytes(workspace, ws_bytes), _stream(stream)))


def qk_decode_step(m, kv, max_batch, max_seq, tokens, pos, B, logits=None, targets=None,
                   logprobs=None, argmax=None, workspace=None, ws_bytes=None, stream=None):
    _check(_load().qk_decode_step(m, _ptr(kv), max_batch, max_seq, _ptr(tokens), _ptr(pos), B,
                                  _ptr(logits), _ptr(targets), _ptr(logprobs), _ptr(argmax),
                                  _ptr(workspace), _nbytes(workspace, ws_bytes), _stream(stream)))


def qk_decode_layer(m, layer, kv, max_batch, max_seq, x, pos, B, workspace=None, ws_bytes=None,
                    stream=None):
    _check(_load().qk_decode_layer(m, layer, _ptr(kv), max_batch, max_seq, _ptr(x), _ptr(pos), B,
                                   _ptr(workspace), _nbytes(workspace, ws_bytes), _stream(stream)))


def qk_score_logprobs(m, tokens, B, T, logprobs, argmax=None, workspace=None, ws_bytes=None,
                      stream=None):
    _check(_load().qk_score_logprobs(m, _ptr(tokens), B, T, _ptr(logprobs), _ptr(argmax),
                                     _ptr(workspace), _nbytes(workspace, ws_bytes),
                                     _stream(stream)))


def qk_grpo_workspace_bytes(B) -> int:
    v = ctypes.c_size_t()
    _check(_load().qk_grpo_workspace_bytes(B, ctypes.byref(v)))
    return v.value


def qk_grpo_token_loss(lp, lp_old, lp_ref, B, T, ld, rewards, group, mask, eps_low, eps_high, beta,
                       loss_tok, loss_mean=None, workspace=None, ws_bytes=None, stream=None):
    _check(_load().qk_grpo_token_loss(_ptr(lp), _ptr(lp_old), _ptr(lp_ref), B, T, ld, _ptr(rewards),
                                      group, _ptr(mask), eps_low, eps_high, beta, _ptr(loss_tok),
                                      _ptr(loss_mean), _ptr(workspace), _nbytes(workspace, ws_bytes),
                                      _stream(stream)))


def qk_grpo_coef(lp, lp_old, lp_ref, B, T, ld, rewards, group, mask, eps_low, eps_high, beta, coef,
                 loss_tok, loss_mean=None, workspace=None, ws_bytes=None, stream=None):
    _check(_load().qk_grpo_coef(_ptr(lp), _ptr(lp_old), _ptr(lp_ref), B, T, ld, _ptr(rewards), group,
                                _ptr(mask), eps_low, eps_high, beta, _ptr(coef), _ptr(loss_tok),
                                _ptr(loss_mean), _ptr(workspace), _nbytes(workspace, ws_bytes),
                                _stream(stream)))


def qk_backward_logprob(m, tokens, B, T, coef, grads, accumulate=0, loss=None, workspace=None,
                        ws_bytes=None, stream=None):
    """grads: a sequence of device fp32 buffers (tensors or addresses), canonical tensor order."""
    arr = (ctypes.c_void_p * len(grads))(*[_ptr(g) for g in grads])
    _check(_load().qk_backward_logprob(m, _ptr(tokens), B, T, _ptr(coef), arr, len(grads), accumulate,
                                       _ptr(loss), _ptr(workspace), _nbytes(workspace, ws_bytes),
                                       _stream(stream)))


def qk_score_grpo(m, tokens, B, T, lp_old, lp_ref, rewards, group, mask, eps_low, eps_high, beta,
                  logprobs, loss_tok, loss_mean=None, workspace=None, ws_bytes=None, stream=None):
    _check(_load().qk_score_grpo(m, _ptr(tokens), B, T, _ptr(lp_old), _ptr(lp_ref), _ptr(rewards),
                                 group, _ptr(mask), eps_low, eps_high, beta, _ptr(logprobs),
                                 _ptr(loss_tok), _ptr(loss_mean), _ptr(workspace),
                                 _nbytes(workspace, ws_bytes), _stream(stream)))


def qk_rollout_teacher_forced(m, kv, max_batch, max_seq, seq, B, P, N, logprobs, argmax=None,
                              workspace=None, ws_bytes=None, stream=None):
    _check(_load().qk_rollout_teacher_forced(m, _ptr(kv), max_batch, max_seq, _ptr(seq), B, P, N,
                                             _ptr(logprobs), _ptr(argmax), _ptr(workspace),
                                             _nbytes(workspace, ws_bytes), _stream(stream)))


def qk_rollout_sampled(m, kv, max_batch, max_seq, prompt, B, P, N, tau, seed, tokens, logprobs,
                       workspace=None, ws_bytes=None, stream=None):
    _check(_load().qk_rollout_sampled(m, _ptr(kv), max_batch, max_seq, _ptr(prompt), B, P, N, tau,
                                      seed, _ptr(tokens), _ptr(logprobs), _ptr(workspace),
                                      _nbytes(workspace, ws_bytes), _stream(stream)))


def qk_prefill_rows(m, kv, max_batch, max_seq, tokens, B, T, start, length=None, last_logits=None,
                    workspace=None, ws_bytes=None, stream=None):
    _check(_load().qk_prefill_rows(m, _ptr(kv), max_batch, max_seq, _ptr(tokens), B, T, _ptr(start),
                                   _ptr(length), _ptr(last_logits), _ptr(workspace),
                                   _nbytes(workspace, ws_bytes), _stream(stream)))


def _pages(table, per_row, n_pages, page_size):
    return qk_kv_pages(_ptr(table), per_row, n_pages, page_size)


def qk_kv_pages_bytes(m, n_pages: int, page_size: int) -> int:
    n = _SZ()
    _check(_load().qk_kv_pages_bytes(m, n_pages, page_size, ctypes.byref(n)))
    return n.value


def qk_decode_step_paged(m, kv, table, per_row, n_pages, page_size, tokens, pos, B, logits=None,
                         targets=None, logprobs=None, argmax=None, workspace=None, ws_bytes=None,
                         stream=None):
    pg = _pages(table, per_row, n_pages, page_size)
    _check(_load().qk_decode_step_paged(m, _ptr(kv), ctypes.byref(pg), _ptr(tokens), _ptr(pos), B,
                                        _ptr(logits), _ptr(targets), _ptr(logprobs), _ptr(argmax),
                                        _ptr(workspace), _nbytes(workspace, ws_bytes), _stream(stream)))


def qk_prefill_rows_paged(m, kv, table, per_row, n_pages, page_size, tokens, B, T, start, length=None,
                          last_logits=None, workspace=None, ws_bytes=None, stream=None):
    pg = _pages(table, per_row, n_pages, page_size)
    _check(_load().qk_prefill_rows_paged(m, _ptr(kv), ctypes.byref(pg), _ptr(tokens), B, T, _ptr(start),
                                         _ptr(length), _ptr(last_logits), _ptr(workspace),
                                         _nbytes(workspace, ws_bytes), _stream(stream)))


def qk_rollout_teacher_forced_paged(m, kv, table, per_row, n_pages, page_size, seq, B, P, N, logprobs,
                                    argmax=None, workspace=None, ws_bytes=None, stream=None):
    pg = _pages(table, per_row, n_pages, page_size)
    _check(_load().qk_rollout_teacher_forced_paged(m, _ptr(kv), ctypes.byref(pg), _ptr(seq), B, P, N,
                                                   _ptr(logprobs), _ptr(argmax), _ptr(workspace),
                                                   _nbytes(workspace, ws_bytes), _stream(stream)))


def qk_rollout_sampled_paged(m, kv, table, per_row, n_pages, page_size, prompt, B, P, N, tau, seed, tokens,
                             logprobs, workspace=None, ws_bytes=None, stream=None):
    pg = _pages(table, per_row, n_pages, page_size)
    _check(_load().qk_rollout_sampled_paged(m, _ptr(kv), ctypes.byref(pg), _ptr(prompt), B, P, N, tau, seed,
                                            _ptr(tokens), _ptr(logprobs), _ptr(workspace),
                                            _nbytes(workspace, ws_bytes), _stream(stream)))


def qk_check_status(m, stream=None) -> int:
    """Returns the status bits (0 when clean); does not raise on QK_EDEVICE or
    QK_ETIMEOUT (the bits say which)."""
    v = ctypes.c_uint32()
    rc = _load().qk_check_status(m, _stream(stream), ctypes.byref(v))
    if rc not in (QK_OK, QK_EDEVICE, QK_ETIMEOUT):
        _check(rc)
    return v.value


def qk_profile_begin(m, kind: int, max_launches: int):
    _check(_load().qk_profile_begin(m, kind, max_launches))


def qk_profile_end(m):
    """Returns (total_ms, launches) of the bracketed kernel class."""
    ms = ctypes.c_float()
    n = _I()
    _check(_load().qk_profile_end(m, ctypes.byref(ms), ctypes.byref(n)))
    return ms.value, n.value


def qk_launch_count() -> int:
    return int(_load().qk_launch_count())


def qk_op_linear(m, A, lda, W, C, ldc, M, N, K, epilogue, scratch=None, scratch_bytes=None,
                 stream=None):
    sb = 0 if scratch is None else _nbytes(scratch, scratch_bytes)
    _check(_load().qk_op_linear(m, _ptr(A), lda, _ptr(W), _ptr(C), ldc, M, N, K, epilogue,
                                _ptr(scratch), sb, _stream(stream)))


def qk_op_linear_swiglu_static(m, A, lda, W, C, ldc, M, N, K, stream=None):
    """SwiGLU linear step with its gate/up intermediate in the library's static device array."""
    _check(_load().qk_op_linear_swiglu_static(m, _ptr(A), lda, _ptr(W), _ptr(C), ldc, M, N, K,
                                              _stream(stream)))


def qk_debug_expire_next_wait(m, wait_cycles: int):
    """Arm the bounded-wait test: the model's next plain tensor-core linear launch
    lets one wait expire after wait_cycles SM cycles (QK_STATUS_TIMEOUT)."""
    _check(_load().qk_debug_expire_next_wait(m, wait_cycles))
