"""ctypes binding of libdvi.so (include/dvi.h): argument marshalling only.

Every step of the decode and update paths runs in the library's CUDA
kernels; PyTorch only provides device memory (weights, workspace, outputs)
and the stream.  Loading fails loudly when libdvi.so has not been built.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libdvi.so")

DVI_F32, DVI_BF16 = 0, 1
STATUS = {0: "DVI_OK", -1: "DVI_ERR_INVALID_ARG", -2: "DVI_ERR_CAPACITY", -3: "DVI_ERR_NONFINITE",
          -4: "DVI_ERR_CUDA", -5: "DVI_ERR_UNIMPLEMENTED", -6: "DVI_ERR_TIMEOUT"}
DEV_BITS = {1: "NONFINITE", 2: "TIMEOUT", 4: "KV_FULL", 8: "BAD_TOKEN", 16: "LOG_FULL"}
BUF = dict(LENS=0, PENDING=1, DRAFT_IDS=2, LOG_U=3, LOG_LOGITS=4, LOG_META=5, GRAD_A=6, GRAD_B=7,
           X_DRAFT=8, X_VERIFY=9, K_CACHE=10, V_CACHE=11, STATUS=12, GRAD_W=13, Z=14)
EXPORTS = ["dvi_workspace_bytes", "dvi_create", "dvi_prefill", "dvi_draft_verify_commit", "dvi_log",
           "dvi_update_drafter", "dvi_ar_step", "dvi_get_stats", "dvi_last_error", "dvi_destroy",
           "dvi_debug_buffer", "dvi_linear", "dvi_timing", "dvi_get_timing", "dvi_linear_noalloc"]


class ModelConfig(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int), ("d_model", ctypes.c_int), ("n_heads", ctypes.c_int),
                ("n_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int), ("d_ffn", ctypes.c_int),
                ("vocab", ctypes.c_int), ("split_k", ctypes.c_int), ("lora_rank", ctypes.c_int),
                ("lora_gamma", ctypes.c_float), ("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float),
                ("dtype", ctypes.c_int)]


class RuntimeConfig(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int), ("k_spec", ctypes.c_int), ("max_seq_len", ctypes.c_int),
                ("log_steps", ctypes.c_int), ("head_mode", ctypes.c_int), ("max_prefill_chunk", ctypes.c_int),
                ("use_graphs", ctypes.c_int), ("bonus", ctypes.c_int), ("persistent", ctypes.c_int),
                ("chain_counters", ctypes.c_int), ("megakernel", ctypes.c_int)]


class LayerWeightsC(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate",
                                               "w_up", "w_down")]


class WeightsC(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("layers", ctypes.POINTER(LayerWeightsC)),
                ("final_norm", ctypes.c_void_p), ("lm_head", ctypes.c_void_p), ("draft_head", ctypes.c_void_p),
                ("lora_a", ctypes.c_void_p), ("lora_b", ctypes.c_void_p)]


class UpdateConfigC(ctypes.Structure):
    _fields_ = [("objective", ctypes.c_int), ("optimizer", ctypes.c_int), ("lr", ctypes.c_float),
                ("beta1", ctypes.c_float), ("beta2", ctypes.c_float), ("adam_eps", ctypes.c_float),
                ("tau", ctypes.c_float), ("lambda0", ctypes.c_float), ("lambda_kl_min", ctypes.c_float),
                ("lambda_pg_max", ctypes.c_float), ("t_warmup", ctypes.c_int), ("t_ramp", ctypes.c_int),
                ("w_ce", ctypes.c_float), ("w_ent", ctypes.c_float), ("w_rl_max", ctypes.c_float),
                ("beta0", ctypes.c_float), ("beta_min", ctypes.c_float), ("t_beta", ctypes.c_float),
                ("baseline_rho", ctypes.c_float), ("keep_grad_w", ctypes.c_int)]


class StatsC(ctypes.Structure):
    _fields_ = [("steps", ctypes.c_int64), ("drafted", ctypes.c_int64), ("accepted", ctypes.c_int64),
                ("committed", ctypes.c_int64), ("updates", ctypes.c_int64), ("kernel_launches", ctypes.c_int64),
                ("last_loss", ctypes.c_float), ("last_kl", ctypes.c_float), ("last_pg", ctypes.c_float),
                ("last_ce", ctypes.c_float), ("last_ent", ctypes.c_float), ("last_rl", ctypes.c_float),
                ("last_kl1", ctypes.c_float), ("last_accept_rate", ctypes.c_float), ("baseline_b", ctypes.c_float),
                ("update_t", ctypes.c_int), ("device_status", ctypes.c_int), ("persistent_ctas", ctypes.c_int),
                ("megakernel_ctas", ctypes.c_int)]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library; raises if it was not built (there is no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with `python -m paper_2510_05421_gb300.build`")
        L = ctypes.CDLL(LIB_PATH)
        vp, i, P = ctypes.c_void_p, ctypes.c_int, ctypes.POINTER
        L.dvi_workspace_bytes.restype = ctypes.c_size_t
        L.dvi_workspace_bytes.argtypes = [P(ModelConfig), P(RuntimeConfig)]
        L.dvi_create.restype = i
        L.dvi_create.argtypes = [P(ModelConfig), P(RuntimeConfig), P(WeightsC), vp, ctypes.c_size_t, vp, P(vp)]
        L.dvi_prefill.restype = i
        L.dvi_prefill.argtypes = [vp, i, vp, i, vp]
        L.dvi_draft_verify_commit.restype = i
        L.dvi_draft_verify_commit.argtypes = [vp, vp, vp, vp]
        L.dvi_log.restype = i
        L.dvi_log.argtypes = [vp, i]
        L.dvi_update_drafter.restype = i
        L.dvi_update_drafter.argtypes = [vp, P(UpdateConfigC)]
        L.dvi_ar_step.restype = i
        L.dvi_ar_step.argtypes = [vp, vp]
        L.dvi_get_stats.restype = i
        L.dvi_get_stats.argtypes = [vp, P(StatsC)]
        L.dvi_last_error.restype = ctypes.c_char_p
        L.dvi_last_error.argtypes = [vp]
        L.dvi_destroy.restype = i
        L.dvi_destroy.argtypes = [vp]
        L.dvi_debug_buffer.restype = i
        L.dvi_debug_buffer.argtypes = [vp, i, P(vp), P(ctypes.c_size_t)]
        L.dvi_linear.restype = i
        L.dvi_linear.argtypes = [vp, vp, i, i, vp, i, vp]
        L.dvi_timing.restype = i
        L.dvi_timing.argtypes = [vp, i]
        L.dvi_get_timing.restype = i
        L.dvi_get_timing.argtypes = [vp, P(ctypes.c_double), P(i)]
        L.dvi_linear_noalloc.restype = i
        L.dvi_linear_noalloc.argtypes = [i, vp, i, i, vp, i, vp, vp]
        _lib = L
    return _lib


class DVIError(RuntimeError):
    pass


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def update_config(h, keep_grad_w: bool = False) -> UpdateConfigC:
    """UpdateConfigC from a workloads.UpdateHyper (or any object with its fields)."""
    obj = {"dvi": 0, "kl": 1, "pg": 2, "ce": 3}[h.objective]
    return UpdateConfigC(obj, 0 if h.optimizer == "adam" else 1, h.lr, h.beta1, h.beta2, h.adam_eps, h.tau,
                         h.lambda0, h.lambda_kl_min, h.lambda_pg_max, h.t_warmup, h.t_ramp, h.w_ce, h.w_ent,
                         h.w_rl_max, h.beta0, h.beta_min, h.t_beta, h.baseline_rho, 1 if keep_grad_w else 0)


@dataclass
class DeviceWeights:
    """Weights resident on the GPU in the model dtype (norm gains, LoRA in f32)."""
    embed: torch.Tensor
    layers: List[Dict[str, torch.Tensor]]
    final_norm: torch.Tensor
    lm_head: torch.Tensor
    draft_head: torch.Tensor
    lora_a: torch.Tensor
    lora_b: torch.Tensor

    @staticmethod
    def from_host(w, dtype: str, device="cuda") -> "DeviceWeights":
        """From workloads.Weights (numpy float32); matrices cast to bf16 or kept f32."""
        td = torch.bfloat16 if dtype == "bf16" else torch.float32

        def mat(a):
            return torch.from_numpy(np.ascontiguousarray(a)).to(device=device).to(td).contiguous()

        def f32(a):
            return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(device=device).contiguous()

        layers = [dict(attn_norm=f32(l.attn_norm), wq=mat(l.wq), wk=mat(l.wk), wv=mat(l.wv), wo=mat(l.wo),
                       ffn_norm=f32(l.ffn_norm), w_gate=mat(l.w_gate), w_up=mat(l.w_up), w_down=mat(l.w_down))
                  for l in w.layers]
        lm = mat(w.lm_head)
        return DeviceWeights(embed=mat(w.embed), layers=layers, final_norm=f32(w.final_norm), lm_head=lm,
                             draft_head=lm.clone(), lora_a=f32(w.lora_a), lora_b=f32(w.lora_b))


def check_linear_noalloc_args(w, x, y) -> None:
    """Raise ValueError unless (w, x, y) is a call dvi_linear_noalloc can run:
    w [N, K] bf16 or f32, x [M, K] f32, y [M, N] f32, all contiguous and on
    one CUDA device, 1 <= M <= 256.  Nothing is launched before this passes,
    so a wrong tensor never reaches the kernel as a raw pointer."""
    if w.dtype not in (torch.bfloat16, torch.float32):
        raise ValueError("linear_noalloc: w must be bf16 or float32")
    if x.dtype != torch.float32 or y.dtype != torch.float32:
        raise ValueError("linear_noalloc: x and y must be float32")
    if len(w.shape) != 2 or len(x.shape) != 2 or len(y.shape) != 2:
        raise ValueError("linear_noalloc: w, x and y must be 2-D")
    n, k = w.shape
    m = x.shape[0]
    if x.shape[1] != k or tuple(y.shape) != (m, n):
        raise ValueError(f"linear_noalloc: shapes w {tuple(w.shape)}, x {tuple(x.shape)}, y {tuple(y.shape)} "
                         "do not match y[M, N] = x[M, K] w[N, K]^T")
    if not 1 <= m <= 256 or n < 1 or k < 1:
        raise ValueError("linear_noalloc: needs 1 <= M <= 256 rows and a non-empty weight")
    if not (w.is_contiguous() and x.is_contiguous() and y.is_contiguous()):
        raise ValueError("linear_noalloc: w, x and y must be contiguous")
    if not (w.is_cuda and x.is_cuda and y.is_cuda) or not (w.device == x.device == y.device):
        raise ValueError("linear_noalloc: w, x and y must be on one CUDA device")


def linear_noalloc(w: torch.Tensor, x: torch.Tensor, y: torch.Tensor, stream=None) -> int:
    """Y = X W^T through dvi_linear_noalloc (no context, no device allocation).

    For callers that cannot allocate device memory: the caller provides w
    ([N, K] bf16 or f32), x ([M, K] f32) and y ([M, N] f32); the library's
    fixed scratch on w's device is used (the call runs with that device
    current).  Raises ValueError on tensors the kernel cannot take; returns
    the library's status code (0 on success).
    """
    check_linear_noalloc_args(w, x, y)
    dtype = DVI_BF16 if w.dtype == torch.bfloat16 else DVI_F32
    with torch.cuda.device(w.device):
        s = stream if stream is not None else torch.cuda.current_stream(w.device)
        return lib().dvi_linear_noalloc(dtype, _ptr(w), w.shape[0], w.shape[1], _ptr(x), x.shape[0], _ptr(y),
                                        ctypes.c_void_p(s.cuda_stream))


class DVIEngine:
    """One DVI context: a layer-split decoder with its KV caches and replay buffer."""

    def __init__(self, shape, dtype: str, weights: DeviceWeights, *, batch: int, k_spec: int, split_k: int,
                 lora_rank: int, lora_gamma: float = 1.0, max_seq_len: int, log_steps: int,
                 prefill_chunk: int = 0, use_graphs: bool = True, device: int = 0, head_mode: int = 0,
                 bonus: bool = False, persistent: bool = False, chain_counters: bool = False,
                 megakernel: bool = True):
        L = lib()
        self.shape, self.dtype, self.w = shape, dtype, weights
        self.B, self.K = batch, k_spec
        self.Kv = k_spec + (1 if bonus else 0)      # verify rows (and committed ids) per sequence
        self.device = torch.device("cuda", device)
        self.cfg = ModelConfig(shape.n_layers, shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim,
                               shape.d_ffn, shape.vocab, split_k, lora_rank, lora_gamma, shape.rms_eps,
                               shape.rope_theta, DVI_BF16 if dtype == "bf16" else DVI_F32)
        self.rt = RuntimeConfig(batch, k_spec, max_seq_len, log_steps, head_mode, prefill_chunk,
                                1 if use_graphs else 0, 1 if bonus else 0, 1 if persistent else 0,
                                1 if chain_counters else 0, 1 if megakernel else 0)
        nbytes = L.dvi_workspace_bytes(ctypes.byref(self.cfg), ctypes.byref(self.rt))
        if nbytes == 0:
            raise DVIError("invalid configuration")
        self.ws = torch.zeros(nbytes + 256, dtype=torch.uint8, device=self.device)
        off = (-self.ws.data_ptr()) % 256
        self.ws_view = self.ws[off:off + nbytes]
        self.stream = torch.cuda.Stream(device=self.device)
        self._layers = (LayerWeightsC * shape.n_layers)(*[
            LayerWeightsC(*[l[n].data_ptr() for n in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate",
                                                     "w_up", "w_down")]) for l in weights.layers])
        self._wc = WeightsC(weights.embed.data_ptr(), self._layers, weights.final_norm.data_ptr(),
                            weights.lm_head.data_ptr(), weights.draft_head.data_ptr(),
                            weights.lora_a.data_ptr() if weights.lora_a.numel() else None,
                            weights.lora_b.data_ptr() if weights.lora_b.numel() else None)
        self.ctx = ctypes.c_void_p()
        torch.cuda.synchronize(self.device)
        rc = L.dvi_create(ctypes.byref(self.cfg), ctypes.byref(self.rt), ctypes.byref(self._wc),
                          ctypes.c_void_p(self.ws_view.data_ptr()), nbytes,
                          ctypes.c_void_p(self.stream.cuda_stream), ctypes.byref(self.ctx))
        if rc != 0:
            raise DVIError(f"dvi_create failed: {STATUS.get(rc, rc)}")
        self.out_ids = torch.zeros(batch, self.Kv, dtype=torch.int32, device=self.device)
        self.n_committed = torch.zeros(batch, dtype=torch.int32, device=self.device)
        self.n_accepted = torch.zeros(batch, dtype=torch.int32, device=self.device)
        self.ar_ids = torch.zeros(batch, dtype=torch.int32, device=self.device)
        self.first = torch.zeros(batch, dtype=torch.int32, device=self.device)
        self.log_steps = log_steps
        self._logging = True        # the library logs by default
        self._logged = 0            # decode steps logged since the last update

    # -- calls ------------------------------------------------------------
    def _check(self, rc, what):
        if rc != 0:
            msg = lib().dvi_last_error(self.ctx).decode()
            raise DVIError(f"{what}: {STATUS.get(rc, rc)} {msg}")

    def prefill(self, seq: int, tokens: torch.Tensor) -> torch.Tensor:
        """Run a device int32 prompt; returns the device tensor of first tokens [B]."""
        if not (tokens.dtype == torch.int32 and tokens.is_cuda and tokens.is_contiguous()):
            raise ValueError("prefill: tokens must be a contiguous int32 CUDA tensor")
        self.stream.wait_stream(torch.cuda.current_stream(self.device))
        rc = lib().dvi_prefill(self.ctx, seq, _ptr(tokens), tokens.numel(),
                               ctypes.c_void_p(self.first.data_ptr() + 4 * seq))
        self._check(rc, "dvi_prefill")
        tokens.record_stream(self.stream)
        return self.first

    def step(self):
        """One draft -> verify -> commit step; device tensors (ids [B,K(+1)], n_committed [B], m [B])
        written on the engine's stream (wait on `self.stream` before reading them elsewhere)."""
        rc = lib().dvi_draft_verify_commit(self.ctx, _ptr(self.out_ids), _ptr(self.n_committed),
                                           _ptr(self.n_accepted))
        self._check(rc, "dvi_draft_verify_commit")
        if self._logging:
            self._logged += 1
        return self.out_ids, self.n_committed, self.n_accepted

    def update(self, hyper, keep_grad_w: bool = False):
        c = hyper if isinstance(hyper, UpdateConfigC) else update_config(hyper, keep_grad_w)
        self._check(lib().dvi_update_drafter(self.ctx, ctypes.byref(c)), "dvi_update_drafter")
        self._logged = 0

    def log(self, enable: bool):
        self._check(lib().dvi_log(self.ctx, 1 if enable else 0), "dvi_log")
        self._logging = bool(enable)

    def ar_step(self) -> torch.Tensor:
        self._check(lib().dvi_ar_step(self.ctx, _ptr(self.ar_ids)), "dvi_ar_step")
        return self.ar_ids

    def stats(self) -> dict:
        s = StatsC()
        self._check(lib().dvi_get_stats(self.ctx, ctypes.byref(s)), "dvi_get_stats")
        d = {f: getattr(s, f) for f, _ in StatsC._fields_}
        d["device_flags"] = [n for b, n in DEV_BITS.items() if s.device_status & b]
        return d

    def linear(self, w: torch.Tensor, x: torch.Tensor) -> torch.Tensor:
        """Y = X W^T through the projection kernel (X float32 [M, K], W [N, K] in the model dtype)."""
        n_out, k_in = w.shape
        y = torch.empty(x.shape[0], n_out, dtype=torch.float32, device=self.device)
        self.stream.wait_stream(torch.cuda.current_stream(self.device))
        self._check(lib().dvi_linear(self.ctx, _ptr(w), n_out, k_in, _ptr(x), x.shape[0], _ptr(y)), "dvi_linear")
        torch.cuda.current_stream(self.device).wait_stream(self.stream)
        return y

    def buffer(self, name: str, dtype: torch.dtype) -> torch.Tensor:
        """A flat view of an internal device buffer (shares memory with the workspace)."""
        p, n = ctypes.c_void_p(), ctypes.c_size_t()
        self._check(lib().dvi_debug_buffer(self.ctx, BUF[name], ctypes.byref(p), ctypes.byref(n)),
                    "dvi_debug_buffer")
        off = p.value - self.ws_view.data_ptr()
        return self.ws_view[off:off + n.value].view(dtype)

    def timing(self, enable: bool):
        self._check(lib().dvi_timing(self.ctx, 1 if enable else 0), "dvi_timing")

    def get_timing(self):
        """{phase: (total ms, calls)} for 'draft', 'verify', 'update' since the last read."""
        ms = (ctypes.c_double * 3)()
        n = (ctypes.c_int * 3)()
        self._check(lib().dvi_get_timing(self.ctx, ms, n), "dvi_get_timing")
        return {k: (ms[i], n[i]) for i, k in enumerate(("draft", "verify", "update"))}

    def sync(self):
        self.stream.synchronize()

    def close(self):
        if self.ctx:
            self.stream.synchronize()
            lib().dvi_destroy(self.ctx)
            self.ctx = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- public generation API -------------------------------------------
    def generate(self, prompts: Sequence[np.ndarray], n_gen: int, update_every: int = 0, hyper=None,
                 max_steps: Optional[int] = None, log: Optional[bool] = None):
        """Self-speculative generation from host prompts to host token lists.

        Each prompt is copied from pinned host memory, prefilled, then steps
        run until every sequence has n_gen tokens; an update of the drafter
        runs after every `update_every` logged steps of the engine (counted
        across calls, so a later call continues the drafter's schedule).
        Replay-buffer logging is on when updates are requested (or when
        `log` says so).  Returns (tokens per
        sequence, per-step accept lengths [steps, B], bytes h2d, bytes d2h).
        """
        self.log(bool(update_every and hyper is not None) if log is None else log)
        h2d = d2h = 0
        for b, p in enumerate(prompts):
            hp = torch.from_numpy(np.ascontiguousarray(p, dtype=np.int32)).pin_memory()
            dp = torch.empty_like(hp, device=self.device)
            with torch.cuda.stream(self.stream):
                dp.copy_(hp, non_blocking=True)
            h2d += hp.numel() * 4
            self.prefill(b, dp)
        first = torch.empty(self.B, dtype=torch.int32).pin_memory()
        with torch.cuda.stream(self.stream):
            first.copy_(self.first, non_blocking=True)
        d2h += self.B * 4
        out_h = torch.empty(self.B, self.Kv, dtype=torch.int32).pin_memory()
        cnt_h = torch.empty(self.B, dtype=torch.int32).pin_memory()
        acc_h = torch.empty(self.B, dtype=torch.int32).pin_memory()
        toks: List[List[int]] = [[] for _ in range(self.B)]
        self.stream.synchronize()
        for b in range(self.B):
            toks[b].append(int(first[b]))
        mats = []
        step = 0
        while min(len(t) for t in toks) < n_gen:
            if max_steps is not None and step >= max_steps:
                break
            ids, cnt, acc = self.step()
            with torch.cuda.stream(self.stream):
                out_h.copy_(ids, non_blocking=True)
                cnt_h.copy_(cnt, non_blocking=True)
                acc_h.copy_(acc, non_blocking=True)
            d2h += (self.B * self.Kv + 2 * self.B) * 4
            self.stream.synchronize()
            for b in range(self.B):
                toks[b].extend(out_h[b, :int(cnt_h[b])].tolist())
            mats.append(acc_h.tolist())
            step += 1
            if update_every and hyper is not None and self._logged >= update_every:
                self.update(hyper)
        return [t[:n_gen] for t in toks], np.array(mats), h2d, d2h

    def generate_ar(self, prompts: Sequence[np.ndarray], n_gen: int):
        """Greedy AR baseline through dvi_ar_step (tokens to host at the end)."""
        outs = torch.empty(self.B, n_gen, dtype=torch.int32, device=self.device)
        for b, p in enumerate(prompts):
            dp = torch.from_numpy(np.ascontiguousarray(p, dtype=np.int32)).to(self.device)
            self.prefill(b, dp)
        with torch.cuda.stream(self.stream):
            outs[:, 0].copy_(self.first)
            for i in range(1, n_gen):
                outs[:, i].copy_(self.ar_step())
        self.stream.synchronize()
        return outs.cpu().numpy()
