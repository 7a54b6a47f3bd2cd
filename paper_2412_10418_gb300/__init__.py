"""GB300 CDSL lookahead step: Python binding of the C ABI in include/cdsl.h.

Argument marshalling only: every step of the path runs in the CUDA library
``libcdsl_gb300.so`` (built in-tree by ``paper_2412_10418_gb300.build``). Importing this module
fails loudly when the library is missing; there is no CPU fallback.

Functions carry the C names (``cdsl_init``, ``cdsl_prefill``, ``cdsl_lookahead``,
``cdsl_verify``, ``cdsl_select``, ``cdsl_step`` ...) and take torch CUDA tensors where the C
call takes device pointers. ``Engine`` bundles a context with its workspace and outputs.
"""
from __future__ import annotations

import ctypes
import os
from typing import List, Optional, Sequence

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libcdsl_gb300.so")

DTYPE_F32, DTYPE_BF16 = 0, 1
STATUS = {0: "CDSL_OK", 1: "CDSL_EINVAL", 2: "CDSL_ENOMEM", 3: "CDSL_ECUDA", 4: "CDSL_ETIMEOUT",
          5: "CDSL_ENONFINITE", 6: "CDSL_ESTATE", 7: "CDSL_ERANGE"}
(CDSL_OK, CDSL_EINVAL, CDSL_ENOMEM, CDSL_ECUDA, CDSL_ETIMEOUT, CDSL_ENONFINITE, CDSL_ESTATE,
 CDSL_ERANGE) = range(8)
S1, S2_S3, S4 = 1, 2, 4


class CdslError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{STATUS.get(code, code)}: {msg}")
        self.code = code


class ModelCfg(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("d_model", ctypes.c_int32),
                ("n_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("d_ffn", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("rope_theta", ctypes.c_float), ("norm_eps", ctypes.c_float)]


class RunCfg(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("k", ctypes.c_int32), ("d", ctypes.c_int32),
                ("max_prompt", ctypes.c_int32), ("max_new", ctypes.c_int32),
                ("n_keywords", ctypes.c_int32), ("a_t", ctypes.c_float), ("r_t", ctypes.c_float),
                ("reward_head", ctypes.c_int32), ("page_size", ctypes.c_int32),
                ("max_chunk", ctypes.c_int32), ("acceptance", ctypes.c_int32),
                ("seed", ctypes.c_uint32), ("step1_budget", ctypes.c_int32)]


_P = ctypes.c_void_p
_I = ctypes.c_int32
EXPORTS = {
    "cdsl_num_weights": (_I, [ctypes.POINTER(ModelCfg)]),
    "cdsl_workspace_size": (_I, [ctypes.POINTER(ModelCfg), ctypes.POINTER(ModelCfg),
                                 ctypes.POINTER(RunCfg), ctypes.POINTER(ctypes.c_size_t)]),
    "cdsl_init": (_I, [ctypes.POINTER(ModelCfg), ctypes.POINTER(_P), ctypes.POINTER(ModelCfg),
                       ctypes.POINTER(_P), ctypes.POINTER(RunCfg), _P, _P, ctypes.c_size_t, _P,
                       ctypes.POINTER(_P)]),
    "cdsl_prefill": (_I, [_P, _P, ctypes.POINTER(ctypes.c_int32), _P]),
    "cdsl_lookahead": (_I, [_P, _P, _P, _P]),
    "cdsl_verify": (_I, [_P, _P, _P, _P, _P]),
    "cdsl_select": (_I, [_P, _P, _P, _P, _P, _P]),
    "cdsl_step": (_I, [_P, _P, _P, _P, _P, _P]),
    "cdsl_get_tokens": (_I, [_P, _P, _P]),
    "cdsl_get_counters": (_I, [_P, ctypes.POINTER(ctypes.c_int64)]),
    "cdsl_get_step1": (_I, [_P, _P, _P, _P]),
    "cdsl_get_status": (_I, [_P, ctypes.POINTER(ctypes.c_int32)]),
    "cdsl_profile": (_I, [_P, _I]),
    "cdsl_get_profile": (_I, [_P, _I, ctypes.POINTER(ctypes.c_double)]),
    "cdsl_get_profile_launches": (_I, [_P, ctypes.POINTER(ctypes.c_double), _I]),
    "cdsl_gemv_noalloc": (_I, [_P, _I, _I, _P, _I, _P, _P]),
    "cdsl_set_wait_limit": (_I, [_P, ctypes.c_uint64]),
    "cdsl_last_error": (ctypes.c_char_p, [_P]),
    "cdsl_destroy": (None, [_P]),
}


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    if not os.path.exists(path):
        raise ImportError(
            f"CUDA library {path} is missing: build it with "
            "`python -m paper_2412_10418_gb300.build` (there is no CPU fallback)")
    lib = ctypes.CDLL(path)
    for name, (res, args) in EXPORTS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib: Optional[ctypes.CDLL] = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        _lib = load_library()
    return _lib


def _ptr(t) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _check(code: int, ctx=None):
    if code != 0:
        msg = lib().cdsl_last_error(ctx)
        raise CdslError(code, msg.decode() if msg else "")


def model_cfg(shape, dtype) -> ModelCfg:
    """ctypes config from any object with the decoder's shape attributes."""
    dt = dtype if isinstance(dtype, int) else (DTYPE_BF16 if dtype == "bf16" else DTYPE_F32)
    return ModelCfg(shape.n_layers, shape.d_model, shape.n_heads, shape.n_kv_heads,
                    shape.head_dim, shape.d_ffn, shape.vocab, dt, shape.rope_theta,
                    shape.norm_eps)


ACCEPT_HARD, ACCEPT_SPECULATIVE = 0, 1


def run_cfg(batch, k, d, max_prompt, max_new, n_keywords, a_t, r_t, reward_head,
            page_size=0, max_chunk=0, acceptance=ACCEPT_HARD, seed=0, step1_budget=0) -> RunCfg:
    return RunCfg(batch, k, d, max_prompt, max_new, n_keywords, a_t, r_t, int(reward_head),
                  page_size, max_chunk, int(acceptance), int(seed) & 0xFFFFFFFF,
                  int(step1_budget))


# ------------------------------------------------------------------------------ C names

def cdsl_num_weights(cfg: ModelCfg) -> int:
    return lib().cdsl_num_weights(ctypes.byref(cfg))


def cdsl_workspace_size(tcfg: ModelCfg, dcfg: ModelCfg, run: RunCfg) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().cdsl_workspace_size(ctypes.byref(tcfg), ctypes.byref(dcfg), ctypes.byref(run),
                                     ctypes.byref(n)))
    return n.value


def cdsl_init(tcfg, t_weights: Sequence, dcfg, d_weights: Sequence, run, reward_head,
              workspace, stream) -> int:
    tw = (_P * len(t_weights))(*[w.data_ptr() for w in t_weights])
    dw = (_P * len(d_weights))(*[w.data_ptr() for w in d_weights])
    ctx = _P(0)
    _check(lib().cdsl_init(ctypes.byref(tcfg), tw, ctypes.byref(dcfg), dw, ctypes.byref(run),
                           _ptr(reward_head), workspace.data_ptr(), workspace.numel(),
                           stream, ctypes.byref(ctx)))
    return ctx.value


def cdsl_prefill(ctx, prompts, prompt_lens: Sequence[int], keywords):
    lens = (ctypes.c_int32 * len(prompt_lens))(*[int(x) for x in prompt_lens])
    _check(lib().cdsl_prefill(ctx, prompts.data_ptr(), lens, keywords.data_ptr()), ctx)


def cdsl_lookahead(ctx, roots=None, draft_tok=None, logq=None):
    _check(lib().cdsl_lookahead(ctx, _ptr(roots), _ptr(draft_tok), _ptr(logq)), ctx)


def cdsl_verify(ctx, logp=None, argmax=None, n_accept=None, logits=None):
    _check(lib().cdsl_verify(ctx, _ptr(logp), _ptr(argmax), _ptr(n_accept), _ptr(logits)), ctx)


def cdsl_select(ctx, beam=None, state=None, emitted=None, n_emitted=None, reward=None):
    _check(lib().cdsl_select(ctx, _ptr(beam), _ptr(state), _ptr(emitted), _ptr(n_emitted),
                             _ptr(reward)), ctx)


def cdsl_step(ctx, beam=None, state=None, emitted=None, n_emitted=None, reward=None):
    _check(lib().cdsl_step(ctx, _ptr(beam), _ptr(state), _ptr(emitted), _ptr(n_emitted),
                           _ptr(reward)), ctx)


def cdsl_get_tokens(ctx, tokens=None, lengths=None):
    _check(lib().cdsl_get_tokens(ctx, _ptr(tokens), _ptr(lengths)), ctx)


def cdsl_get_counters(ctx) -> List[int]:
    out = (ctypes.c_int64 * 8)()
    _check(lib().cdsl_get_counters(ctx, out), ctx)
    return list(out)


def cdsl_get_step1(ctx, need=None, tokens=None, reward=None):
    _check(lib().cdsl_get_step1(ctx, _ptr(need), _ptr(tokens), _ptr(reward)), ctx)


def cdsl_set_wait_limit(ctx, ns: int):
    """Limit (nanoseconds) of the tensor-core kernels' bounded waits; see include/cdsl.h."""
    _check(lib().cdsl_set_wait_limit(ctx, int(ns)), ctx)


def cdsl_get_status(ctx) -> int:
    v = ctypes.c_int32(0)
    _check(lib().cdsl_get_status(ctx, ctypes.byref(v)), ctx)
    return v.value


PROFILE_OFF, PROFILE_EVENTS, PROFILE_IN_GRAPH = 0, 1, 2


def cdsl_profile(ctx, mode):
    """mode 0 off, 1 CUDA events around direct launches, 2 in-graph stamps (see cdsl.h);
    True / False stand for 1 / 0."""
    _check(lib().cdsl_profile(ctx, int(mode)), ctx)


GEMM_IMPLS = {0: "gemm_simt", 1: "gemv_stream", 2: "gemm_tc"}
KERNEL_CLASSES = {0: "gemm_simt", 1: "gemv_stream", 2: "gemm_tc", 3: "attention", 4: "rmsnorm",
                  5: "row_stats", 6: "embed", 7: "step_logic"}
STAMPED_STEPS = 8   # cdsl_get_profile class of the stamped steps themselves (mode 2)


def cdsl_get_profile(ctx, impl: int):
    out = (ctypes.c_double * 4)()
    _check(lib().cdsl_get_profile(ctx, impl, out), ctx)
    return dict(launches=int(out[0]), ms=out[1], bytes=out[2], flops=out[3])


def cdsl_get_profile_launches(ctx, capacity: int = 8192):
    """Per-launch timing records [(class, ms, bytes, flops)] in launch order."""
    out = (ctypes.c_double * (4 * capacity))()
    n = lib().cdsl_get_profile_launches(ctx, out, capacity)
    if n < 0:
        raise CdslError(-n, cdsl_last_error(ctx))
    return [(int(out[4 * i]), out[4 * i + 1], out[4 * i + 2], out[4 * i + 3]) for i in range(n)]


def cdsl_gemv_noalloc(w, x, y, stream=None):
    """y[R, N] = x[R, K] w^T through the weight-streaming kernel with its scratch in a fixed
    array inside the library (no device memory is allocated); see include/cdsl.h.

    The C ABI sees only pointers and sizes, so the shapes, dtypes, layouts and devices are
    checked here: w bfloat16 [N, K], x float32 [R, K], y float32 [R, N], all contiguous and on
    the current CUDA device. Anything else raises CdslError(CDSL_EINVAL) before the call."""
    import torch

    def bad(why):
        raise CdslError(CDSL_EINVAL, "cdsl_gemv_noalloc: " + why)

    ts = (w, x, y)
    if not all(isinstance(t, torch.Tensor) for t in ts):
        bad("w, x and y must be torch tensors")
    if w.dtype != torch.bfloat16 or x.dtype != torch.float32 or y.dtype != torch.float32:
        bad("w must be bfloat16, x and y float32")
    if w.dim() != 2 or x.dim() != 2 or y.dim() != 2:
        bad("w, x and y must be 2-D")
    N, K = w.shape
    R = x.shape[0]
    if tuple(x.shape) != (R, K) or tuple(y.shape) != (R, N):
        bad(f"shapes: w {tuple(w.shape)}, x {tuple(x.shape)}, y {tuple(y.shape)} "
            "(want [N, K], [R, K], [R, N])")
    if not all(t.is_contiguous() for t in ts):
        bad("w, x and y must be contiguous")
    dev = torch.cuda.current_device() if torch.cuda.is_available() else None
    if not all(t.is_cuda and t.device.index == dev for t in ts):
        bad("w, x and y must be on the current CUDA device")
    _check(lib().cdsl_gemv_noalloc(w.data_ptr(), N, K, x.data_ptr(), R, y.data_ptr(), stream))


def cdsl_last_error(ctx=None) -> str:
    m = lib().cdsl_last_error(ctx)
    return m.decode() if m else ""


def cdsl_destroy(ctx):
    lib().cdsl_destroy(ctx)


# ------------------------------------------------------------------------------ Engine

class Engine:
    """A context plus its workspace and per-step output tensors (all on one CUDA device).

    target_weights / draft_weights: torch tensors in the C ABI order (cdsl_num_weights of
    them), kept referenced for the engine's lifetime."""

    def __init__(self, target_shape, draft_shape, dtype, target_weights, draft_weights, *,
                 batch, k, d, max_prompt, max_new, n_keywords, a_t, r_t, reward_head=None,
                 page_size=0, max_chunk=0, acceptance=ACCEPT_HARD, seed=0, step1_budget=0,
                 stream=None, device="cuda"):
        import torch

        self.torch = torch
        self.tcfg = model_cfg(target_shape, dtype)
        self.dcfg = model_cfg(draft_shape, dtype)
        self.run = run_cfg(batch, k, d, max_prompt, max_new, n_keywords, a_t, r_t,
                           reward_head is not None, page_size, max_chunk, acceptance, seed,
                           step1_budget)
        self.B, self.k, self.d, self.V = batch, k, d, target_shape.vocab
        self.max_prompt, self.max_new = max_prompt, max_new
        self.tw, self.dw = list(target_weights), list(draft_weights)
        self.head = reward_head
        self.stream = stream if stream is not None else torch.cuda.Stream(device=device)
        nbytes = cdsl_workspace_size(self.tcfg, self.dcfg, self.run)
        self.ws = torch.empty(nbytes, dtype=torch.uint8, device=device)
        self.ctx = cdsl_init(self.tcfg, self.tw, self.dcfg, self.dw, self.run, self.head, self.ws,
                             self.stream.cuda_stream)
        i32, f32 = torch.int32, torch.float32
        B, K, D = batch, k, d
        z = lambda *s, dt=i32: torch.zeros(s, dtype=dt, device=device)
        self.roots, self.draft_tok, self.logq = z(B, K), z(B, K, D), z(B, K, D, dt=f32)
        self.logp, self.argmax, self.n_accept = z(B, K, D, dt=f32), z(B, K, D + 1), z(B, K)
        self.beam, self.state, self.emitted = z(B), z(B), z(B, D + 1)
        self.n_emitted, self.reward = z(B), z(B, K, 2, dt=f32)

    def prefill(self, prompts, prompt_lens, keywords):
        with self.torch.cuda.stream(self.stream):
            self._prompts = prompts.to(self.ws.device, self.torch.int32).contiguous()
            self._kw = keywords.to(self.ws.device, self.torch.int32).contiguous()
        self.stream.synchronize()
        cdsl_prefill(self.ctx, self._prompts, prompt_lens, self._kw)

    def lookahead(self):
        cdsl_lookahead(self.ctx, self.roots, self.draft_tok, self.logq)

    def verify(self, logits=None):
        cdsl_verify(self.ctx, self.logp, self.argmax, self.n_accept, logits)

    def select(self):
        cdsl_select(self.ctx, self.beam, self.state, self.emitted, self.n_emitted, self.reward)

    def step(self):
        cdsl_step(self.ctx, self.beam, self.state, self.emitted, self.n_emitted, self.reward)

    def tokens(self):
        t = self.torch.empty((self.B, self.max_prompt + self.max_new), dtype=self.torch.int32,
                             device=self.ws.device)
        n = self.torch.empty(self.B, dtype=self.torch.int32, device=self.ws.device)
        cdsl_get_tokens(self.ctx, t, n)
        self.stream.synchronize()
        return t, n

    def step1(self):
        """Step-1 round 2 of the last select / step (budget 2): need [B], tokens [B, d+1]
        (x', lh_1..lh_d), reward [B]."""
        t = self.torch
        need = t.zeros(self.B, dtype=t.int32, device=self.ws.device)
        tok = t.zeros((self.B, self.d + 1), dtype=t.int32, device=self.ws.device)
        rew = t.zeros(self.B, dtype=t.float32, device=self.ws.device)
        cdsl_get_step1(self.ctx, need, tok, rew)
        self.stream.synchronize()
        return need, tok, rew

    def counters(self):
        return cdsl_get_counters(self.ctx)

    def status(self):
        return cdsl_get_status(self.ctx)

    def close(self):
        if getattr(self, "ctx", None):
            cdsl_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
