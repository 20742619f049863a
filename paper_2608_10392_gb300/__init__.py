"""GB300 (sm_103a) UniF-MoE layer forward pass: thin ctypes binding of the
C ABI in include/unif_moe.h.

Every step of the forward runs inside libunif_moe.so; this module only
marshals torch tensors (device memory, streams) into the C calls. There is no
fallback: if the library is missing, importing `lib()` raises.

    layer = Layer(d_model=384, d_ff=1536, n_experts=8, n_blocks=8, dtype="bf16",
                  max_tokens=12608)
    layer.load_weights(w_router, w_up, w_down)          # CUDA tensors
    y = layer.forward(x)                                # x [T][d] CUDA tensor
"""
from __future__ import annotations

import ctypes as C
import math
import os
from typing import Optional

import torch

__all__ = ["Layer", "lib", "UnifMoeError", "ERR", "EXPORTS", "Options", "FEATURE_NORM_FIRST",
           "FEATURE_HOST_IO", "FEATURE_BACKWARD", "FEATURE_DIAGNOSTICS", "FEATURES_DEFAULT",
           "FEATURES_ALL"]

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "lib", "libunif_moe.so")

ERR = {0: "OK", -1: "ERR_ARG", -2: "ERR_SHAPE", -3: "ERR_CAPACITY", -4: "ERR_CUDA",
       -5: "ERR_TIMEOUT", -6: "ERR_STATE"}

# Every symbol include/unif_moe.h declares.
EXPORTS = ["unif_moe_default_thresholds", "unif_moe_default_options", "unif_moe_create",
           "unif_moe_create_ex", "unif_moe_load_weights",
           "unif_moe_load_upcycled", "unif_moe_forward", "unif_moe_sublayer_forward",
           "unif_moe_backward", "unif_moe_value_alignment", "unif_moe_functional_demand",
           "unif_moe_forward_host", "unif_moe_forward_host_async",
           "unif_moe_forward_host_wait", "unif_moe_get_routing",
           "unif_moe_get_groups", "unif_moe_max_rows", "unif_moe_pass_tokens",
           "unif_moe_kernels_per_forward",
           "unif_moe_set_stage_events",
           "unif_moe_sync_status", "unif_moe_selftest_timeout", "unif_moe_group_noalloc",
           "unif_moe_destroy", "unif_moe_last_error"]


class UnifMoeError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__("%s (%d): %s" % (ERR.get(code, "?"), code, msg))
        self.code = code


class Thresholds(C.Structure):
    _fields_ = [("tau", C.c_float), ("alpha_fixed", C.c_float), ("beta_fixed", C.c_float),
                ("topk_fixed", C.c_int), ("prefix_blocks", C.c_int)]


class Options(C.Structure):
    _fields_ = [("features", C.c_uint), ("gemm_kernels", C.c_int)]


FEATURE_NORM_FIRST, FEATURE_HOST_IO, FEATURE_BACKWARD, FEATURE_DIAGNOSTICS = 1, 2, 4, 8
FEATURES_DEFAULT, FEATURES_ALL = 3, 15
GEMM_KERNELS = {"auto": 0, "streaming": 1, "grouped": 2, "expert_tile": 3}


_lib = None


def lib(path: str = LIB_PATH) -> C.CDLL:
    """Loads libunif_moe.so (built by __graft_entry__.build()); raises if absent."""
    global _lib
    if _lib is None:
        if not os.path.exists(path):
            raise RuntimeError("libunif_moe.so not built (%s); run __graft_entry__.build()" % path)
        L = C.CDLL(path)
        P, I = C.c_void_p, C.c_int
        L.unif_moe_default_thresholds.argtypes = [C.POINTER(Thresholds)]
        L.unif_moe_default_thresholds.restype = None
        L.unif_moe_create.argtypes = [C.POINTER(P), I, I, I, I, C.POINTER(Thresholds), I, I]
        L.unif_moe_default_options.argtypes = [C.POINTER(Options)]
        L.unif_moe_default_options.restype = None
        L.unif_moe_create_ex.argtypes = [C.POINTER(P), I, I, I, I, C.POINTER(Thresholds), I, I,
                                         C.POINTER(Options)]
        L.unif_moe_load_weights.argtypes = [P, P, P, P, P, P]
        L.unif_moe_forward.argtypes = [P, P, P, I, P, P, P, P]
        L.unif_moe_load_upcycled.argtypes = [P, P, P, P, P, P]
        L.unif_moe_sublayer_forward.argtypes = [P, P, P, I, P, P, P, P, P, C.c_float, I, P]
        L.unif_moe_backward.argtypes = [P, P, P, I, P, P, P, P, P, P, C.c_float, P, P]
        L.unif_moe_value_alignment.argtypes = [P, C.c_float, P, P]
        L.unif_moe_functional_demand.argtypes = [P, P, I, P, C.c_float, C.c_float, P, P, P, P]
        L.unif_moe_forward_host.argtypes = [P, P, P, I, P, P, P, P]
        L.unif_moe_forward_host_async.argtypes = [P, P, P, I, P, P, P, P]
        L.unif_moe_forward_host_wait.argtypes = [P]
        L.unif_moe_get_routing.argtypes = [P, P, P, P, P, P, P]
        L.unif_moe_get_groups.argtypes = [P, P, P, P, P, C.POINTER(C.c_int64), P]
        L.unif_moe_max_rows.argtypes = [P]
        L.unif_moe_max_rows.restype = C.c_int64
        L.unif_moe_pass_tokens.argtypes = [P]
        L.unif_moe_kernels_per_forward.argtypes = [P]
        L.unif_moe_set_stage_events.argtypes = [P, P]
        L.unif_moe_sync_status.argtypes = [P, P]
        L.unif_moe_selftest_timeout.argtypes = [P, I, P]
        L.unif_moe_group_noalloc.argtypes = [I, I, I] + [P] * 11 + [C.c_int64, P]
        L.unif_moe_destroy.argtypes = [P]
        L.unif_moe_destroy.restype = None
        L.unif_moe_last_error.restype = C.c_char_p
        for name in EXPORTS:
            if name not in ("unif_moe_default_thresholds", "unif_moe_default_options",
                            "unif_moe_destroy",
                            "unif_moe_last_error", "unif_moe_max_rows"):
                getattr(L, name).restype = C.c_int
        _lib = L
    return _lib


def _check(rc: int):
    if rc != 0:
        raise UnifMoeError(rc, lib().unif_moe_last_error().decode())


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else stream


class Layer:
    """One UniF-MoE layer (Sec. III): K residual experts plus one shared
    expert, FFN width H split into B blocks. dtype "bf16" (tensor cores) or
    "f32" (CUDA-core FMA). `features` (FEATURE_* bits) picks the optional
    workspaces allocated at create time; `gemm_kernels` "grouped" ((expert,
    block) groups, weight-stationary kernels where they fit), "streaming"
    ((expert, block) groups, streaming kernels), "expert_tile" (rows grouped
    by expert, both projections in one kernel, where it applies) or "auto"
    (expert_tile where it applies, else grouped)."""

    def __init__(self, d_model: int, d_ff: int, n_experts: int, n_blocks: int,
                 dtype: str = "bf16", max_tokens: int = 65536, tau: float = math.nan,
                 alpha_fixed: float = math.nan, beta_fixed: float = math.nan,
                 topk_fixed: int = 0, prefix_blocks: int = 0, features: int = FEATURES_DEFAULT,
                 gemm_kernels: str = "auto"):
        self.d, self.H, self.K, self.B = d_model, d_ff, n_experts, n_blocks
        self.dtype = dtype
        self.torch_dtype = torch.bfloat16 if dtype == "bf16" else torch.float32
        self.max_tokens = max_tokens
        th = Thresholds(tau, alpha_fixed, beta_fixed, topk_fixed, prefix_blocks)
        opts = Options(features, GEMM_KERNELS[gemm_kernels])
        h = C.c_void_p()
        _check(lib().unif_moe_create_ex(C.byref(h), d_model, d_ff, n_experts, n_blocks,
                                        C.byref(th), 1 if dtype == "bf16" else 0, max_tokens,
                                        C.byref(opts)))
        self._h = h
        self.last_T = 0

    def close(self):
        if getattr(self, "_h", None) is not None and self._h.value:
            lib().unif_moe_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def load_weights(self, w_router: torch.Tensor, w_up: torch.Tensor, w_down: torch.Tensor,
                     router_bias: Optional[torch.Tensor] = None, stream=None):
        for t in (w_router, w_up, w_down):
            assert t.is_cuda and t.dtype == self.torch_dtype and t.is_contiguous()
        if router_bias is not None:
            assert router_bias.is_cuda and router_bias.dtype == torch.float32
        self._keep = (w_router, w_up, w_down, router_bias)  # alive until the copy ran
        _check(lib().unif_moe_load_weights(self._h, _ptr(w_router), _ptr(w_up), _ptr(w_down),
                                           _ptr(router_bias), _stream(stream)))

    def load_upcycled(self, w_router: torch.Tensor, w_up_dense: torch.Tensor,
                      w_down_dense: torch.Tensor, router_bias: Optional[torch.Tensor] = None,
                      stream=None):
        """Every expert starts as the dense FFN (w_up_dense [H][d], w_down_dense [d][H])."""
        for t in (w_router, w_up_dense, w_down_dense):
            assert t.is_cuda and t.dtype == self.torch_dtype and t.is_contiguous()
        if router_bias is not None:
            assert router_bias.is_cuda and router_bias.dtype == torch.float32
        self._keep = (w_router, w_up_dense, w_down_dense, router_bias)
        _check(lib().unif_moe_load_upcycled(self._h, _ptr(w_router), _ptr(w_up_dense),
                                            _ptr(w_down_dense), _ptr(router_bias),
                                            _stream(stream)))

    def sublayer_forward(self, x: torch.Tensor, ln_gamma: torch.Tensor, ln_beta: torch.Tensor,
                         eps: float, norm_first: bool, out: Optional[torch.Tensor] = None,
                         mask: Optional[torch.Tensor] = None,
                         shared_counts: Optional[torch.Tensor] = None,
                         residual_counts: Optional[torch.Tensor] = None,
                         stream=None) -> torch.Tensor:
        """x + F(LN(x)) (norm_first) or LN(x + F(x)), F this layer."""
        T = x.shape[0]
        if out is None:
            out = torch.empty_like(x)
        _check(lib().unif_moe_sublayer_forward(self._h, _ptr(x), _ptr(out), T, _ptr(mask),
                                               _ptr(shared_counts), _ptr(residual_counts),
                                               _ptr(ln_gamma), _ptr(ln_beta), float(eps),
                                               1 if norm_first else 0, _stream(stream)))
        self.last_T = T
        return out

    def forward(self, x: torch.Tensor, out: Optional[torch.Tensor] = None,
                mask: Optional[torch.Tensor] = None, shared_counts: Optional[torch.Tensor] = None,
                residual_counts: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
        T = x.shape[0]
        if out is None:
            out = torch.empty_like(x)
        _check(lib().unif_moe_forward(self._h, _ptr(x), _ptr(out), T, _ptr(mask),
                                      _ptr(shared_counts), _ptr(residual_counts),
                                      _stream(stream)))
        self.last_T = T
        return out

    def backward(self, x: torch.Tensor, dy: torch.Tensor, mask: Optional[torch.Tensor] = None,
                 lambda_div: float = 0.0, want_bias: bool = False, out: Optional[dict] = None,
                 stream=None) -> dict:
        """Gradients of the last forward (which must have run on x) given
        dL/dy (Sec. III-E): dict of fp32 CUDA tensors dx, dw_up, dw_down,
        dw_router (plus lambda_div dL_div/dW*), dbias (want_bias), l_div;
        `out`, such a dict from an earlier call, is filled again."""
        T = x.shape[0]
        dev = x.device
        f32 = dict(dtype=torch.float32, device=dev)
        g = out if out is not None else dict(
            dx=torch.empty(T, self.d, **f32),
            dw_up=torch.empty(self.K + 1, self.H, self.d, **f32),
            dw_down=torch.empty(self.K + 1, self.d, self.H, **f32),
            dw_router=torch.empty(self.d, self.K + 1, **f32),
            dbias=torch.empty(self.K + 1, **f32) if want_bias else None,
            l_div=torch.empty(1, **f32))
        _check(lib().unif_moe_backward(self._h, _ptr(x), _ptr(dy), T, _ptr(mask), _ptr(g["dx"]),
                                       _ptr(g["dw_up"]), _ptr(g["dw_down"]),
                                       _ptr(g["dw_router"]), _ptr(g["dbias"]),
                                       float(lambda_div), _ptr(g["l_div"]), _stream(stream)))
        return g

    def value_alignment(self, delta: float, stream=None) -> torch.Tensor:
        """rho [K][K] of the residual experts (Sec. II-B, Eq. shared-set)."""
        rho = torch.empty(self.K, self.K, dtype=torch.float32, device=torch.device("cuda"))
        _check(lib().unif_moe_value_alignment(self._h, float(delta), _ptr(rho), _stream(stream)))
        return rho

    def functional_demand(self, x: torch.Tensor, w_res: torch.Tensor, delta: float, eps: float,
                          stream=None) -> dict:
        """k_eps [T], e [T][K] and the top-2 pair [T][2] of every token (Sec.
        II-B); w_res [d][K] the residual router (layer dtype)."""
        T = x.shape[0]
        dev = x.device
        out = dict(k_eps=torch.empty(T, dtype=torch.int32, device=dev),
                   err=torch.empty(T, self.K, dtype=torch.float32, device=dev),
                   pair=torch.empty(T, 2, dtype=torch.int32, device=dev))
        _check(lib().unif_moe_functional_demand(self._h, _ptr(x), T, _ptr(w_res), float(delta),
                                                float(eps), _ptr(out["k_eps"]), _ptr(out["err"]),
                                                _ptr(out["pair"]), _stream(stream)))
        return out

    def forward_host(self, x_host: torch.Tensor, out_host: torch.Tensor,
                     mask_host: Optional[torch.Tensor] = None,
                     shared_counts_host: Optional[torch.Tensor] = None,
                     residual_counts_host: Optional[torch.Tensor] = None, stream=None):
        T = x_host.shape[0]
        _check(lib().unif_moe_forward_host(self._h, _ptr(x_host), _ptr(out_host), T,
                                           _ptr(mask_host), _ptr(shared_counts_host),
                                           _ptr(residual_counts_host), _stream(stream)))
        self.last_T = T
        return out_host

    def forward_host_async(self, x_host: torch.Tensor, out_host: torch.Tensor,
                           mask_host: Optional[torch.Tensor] = None,
                           shared_counts_host: Optional[torch.Tensor] = None,
                           residual_counts_host: Optional[torch.Tensor] = None, stream=None):
        """Enqueues a forward of host tensors and returns at once (the copies
        overlap other calls' kernels); results are in out_host (and the
        counts) after forward_host_wait()."""
        T = x_host.shape[0]
        _check(lib().unif_moe_forward_host_async(self._h, _ptr(x_host), _ptr(out_host), T,
                                                 _ptr(mask_host), _ptr(shared_counts_host),
                                                 _ptr(residual_counts_host), _stream(stream)))
        self.last_T = T
        return out_host

    def forward_host_wait(self):
        _check(lib().unif_moe_forward_host_wait(self._h))

    def routing(self, stream=None) -> dict:
        """Decisions of the last forward, as CUDA tensors."""
        T, K = self.last_T, self.K
        dev = torch.device("cuda")
        r = dict(alpha=torch.empty(T, dtype=torch.float32, device=dev),
                 shared_mask=torch.empty(T, dtype=torch.int64, device=dev),
                 expert_mask=torch.empty(T, dtype=torch.int64, device=dev),
                 q=torch.empty(T, K, dtype=torch.int32, device=dev),
                 p=torch.empty(T, K, dtype=torch.float32, device=dev))
        _check(lib().unif_moe_get_routing(self._h, _ptr(r["alpha"]), _ptr(r["shared_mask"]),
                                          _ptr(r["expert_mask"]), _ptr(r["q"]), _ptr(r["p"]),
                                          _stream(stream)))
        return r

    def max_rows(self) -> int:
        return int(lib().unif_moe_max_rows(self._h))

    def pass_tokens(self) -> int:
        """Tokens per pass: larger forwards run in passes of this many tokens."""
        return int(lib().unif_moe_pass_tokens(self._h))

    def kernels_per_forward(self) -> int:
        return int(lib().unif_moe_kernels_per_forward(self._h))

    def groups(self, stream=None):
        """Group table of the last forward (host tensors): counts [G],
        offsets [G+1], row tokens and weights [offsets[G]]."""
        G = (self.K + 1) * self.B
        n = self.max_rows()
        counts = torch.empty(G, dtype=torch.int32)
        offsets = torch.empty(G + 1, dtype=torch.int32)
        tok = torch.empty(n, dtype=torch.int32)
        w = torch.empty(n, dtype=torch.float32)
        nrows = C.c_int64()
        _check(lib().unif_moe_get_groups(self._h, _ptr(counts), _ptr(offsets), _ptr(tok), _ptr(w),
                                         C.byref(nrows), _stream(stream)))
        return counts, offsets, tok[:nrows.value].clone(), w[:nrows.value].clone()

    def set_stage_events(self, events):
        """events: 6 torch.cuda.Event(enable_timing=True) already recorded once
        (so that the CUDA event exists), or None to stop stage timing."""
        if events is None:
            _check(lib().unif_moe_set_stage_events(self._h, None))
            return
        arr = (C.c_void_p * 6)(*[e.cuda_event for e in events])
        self._events = events
        _check(lib().unif_moe_set_stage_events(self._h, arr))

    def sync_status(self, stream=None) -> int:
        return lib().unif_moe_sync_status(self._h, _stream(stream))

    def selftest_timeout(self, timeout_us: int, stream=None):
        _check(lib().unif_moe_selftest_timeout(self._h, timeout_us, _stream(stream)))
