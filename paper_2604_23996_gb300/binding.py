"""ctypes binding of the SMoES C ABI (include/smoes.h).

Argument marshalling only: every computation runs in ``lib/libsmoes.so``. Functions carry the
C names; tensors are passed as torch CUDA tensors (their data pointers) or None. Importing this
module fails loudly when the library has not been built: there is no fallback path.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Optional

import numpy as np
import torch

from .build import LIB

if not os.path.exists(LIB):
    raise ImportError(f"SMoES CUDA library not built ({LIB}); run __graft_entry__.build()")
_lib = C.CDLL(LIB)

SMOES_OK = 0
STATUS_NAMES = {0: "SMOES_OK", -1: "SMOES_ERR_INVALID_ARG", -2: "SMOES_ERR_UNSUPPORTED",
                -3: "SMOES_ERR_ALIGNMENT", -4: "SMOES_ERR_WORKSPACE", -5: "SMOES_ERR_CUDA",
                -6: "SMOES_ERR_DEVICE_TIMEOUT", -7: "SMOES_ERR_DATA"}
SMOES_F32, SMOES_BF16 = 0, 1
SMOES_GATE_SOFTMAX, SMOES_GATE_SIGMOID = 0, 1
SMOES_SCORE_PROVIDED, SMOES_SCORE_GAUSS, SMOES_SCORE_ATTN, SMOES_SCORE_GMM = 0, 1, 2, 3
(SMOES_CALL_ROUTER_FWD, SMOES_CALL_ROUTER_FWD_PERMUTE, SMOES_CALL_ROUTER_BWD, SMOES_CALL_BIN_PERMUTE,
 SMOES_CALL_ATTN_SCORE) = 0, 1, 2, 3, 4


class SmoesError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: {STATUS_NAMES.get(code, code)} ({smoes_status_string(code)})")
        self.code = code


class RouterDesc(C.Structure):
    _fields_ = [("T", C.c_int), ("d", C.c_int), ("E", C.c_int), ("k", C.c_int),
                ("n_bins", C.c_int), ("n_samples", C.c_int), ("dtype", C.c_int),
                ("sample_offsets_host", C.POINTER(C.c_int32)),
                ("expert_bin_host", C.POINTER(C.c_int32)), ("renorm_topk", C.c_int),
                ("attn_max_heads", C.c_int), ("gate", C.c_int), ("score_bias", C.c_void_p),
                ("mi_topk_mask", C.c_int)]


class GaussArgs(C.Structure):
    _fields_ = [("X", C.c_void_p), ("mu", C.c_void_p), ("var", C.c_void_p), ("tau", C.c_float)]


class AttnArgs(C.Structure):
    _fields_ = [("Q", C.c_void_p), ("K", C.c_void_p), ("B", C.c_int), ("H", C.c_int),
                ("S", C.c_int), ("hd", C.c_int), ("is_vision", C.c_void_p), ("m_prev", C.c_void_p),
                ("key_bias", C.c_void_p), ("sm_scale", C.c_float), ("causal", C.c_int),
                ("xattn_norm", C.c_void_p), ("x_norm", C.c_void_p)]


class GmmArgs(C.Structure):
    _fields_ = [("X", C.c_void_p), ("n_components", C.c_int), ("log_pi", C.c_void_p),
                ("mu", C.c_void_p), ("var", C.c_void_p), ("tau", C.c_float)]


class ScoreArgs(C.Structure):
    _fields_ = [("gauss", GaussArgs), ("attn", AttnArgs), ("gmm", GmmArgs)]


_vp, _i, _f, _sz = C.c_void_p, C.c_int, C.c_float, C.c_size_t
_sig = {
    "smoes_plan_create": (_i, [C.POINTER(RouterDesc), C.POINTER(_vp)]),
    "smoes_plan_destroy": (None, [_vp]),
    "smoes_workspace_bytes": (_sz, [_vp]),
    "smoes_workspace_init": (_i, [_vp, _vp, _sz, _vp]),
    "smoes_status_string": (C.c_char_p, [_i]),
    "smoes_plan_set_wait_limit": (_i, [_vp, C.c_uint64]),
    "smoes_call_launches": (_i, [_vp, _i]),
    "smoes_read_device_status": (_i, [_vp, _vp, _vp, C.POINTER(C.c_int32)]),
    "smoes_modality_score": (_i, [_vp, _i, C.POINTER(ScoreArgs), _vp, _vp, _sz, _vp]),
    "smoes_router_fwd": (_i, [_vp, _vp, _vp, _vp, C.POINTER(GaussArgs), _vp, _vp, _vp, _vp, _vp,
                              _vp, _vp, _vp, _sz, _vp]),
    "smoes_router_fwd_permute": (_i, [_vp, _vp, _vp, _vp, C.POINTER(GaussArgs), _vp, _vp, _vp, _vp,
                                      _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz,
                                      _vp]),
    "smoes_router_bwd": (_i, [_vp, _vp, _vp, _vp, _vp, _vp, _f, _vp, _i, _vp, _vp, _vp, _sz, _vp]),
    "smoes_bin_permute": (_i, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "smoes_bin_permute_noalloc": (_i, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp]),
    "smoes_gaussian_stats_update": (_i, [_vp, _vp, _vp, C.c_double, _vp, _vp, _vp, _vp, _vp, _vp,
                                         _sz, _vp]),
    "smoes_adaptive_bins": (_i, [_vp, _vp, C.c_double, _vp, _vp, _vp, _vp]),
    "smoes_bin_balance": (_i, [_vp, _vp, _f, _vp, _vp, _vp, _vp, _sz, _vp]),
    "smoes_attention_fwd": (_i, [_vp, C.POINTER(AttnArgs), _vp, _i, _vp, _vp, _vp, _sz, _vp]),
}
for _name, (_res, _args) in _sig.items():
    _fn = getattr(_lib, _name)
    _fn.restype = _res
    _fn.argtypes = _args


def exported_symbols():
    return list(_sig)


def _p(t: Optional[torch.Tensor]):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(stream=None):
    if stream is None:
        stream = torch.cuda.current_stream()
    return C.c_void_p(stream.cuda_stream)


def _check(code: int, what: str):
    if code != SMOES_OK:
        raise SmoesError(code, what)


def smoes_status_string(code: int) -> str:
    return _lib.smoes_status_string(code).decode()


def smoes_plan_create(T, d, E, k, n_bins, sample_offsets, expert_bin, dtype, renorm_topk=0,
                      attn_max_heads=0, gate=0, score_bias=None, mi_topk_mask=0):
    """Returns (status, plan handle). sample_offsets [B+1] and expert_bin [E] are host arrays."""
    offs = np.ascontiguousarray(np.asarray(sample_offsets, dtype=np.int32))
    eb = np.ascontiguousarray(np.asarray(expert_bin, dtype=np.int32))
    desc = RouterDesc(T, d, E, k, n_bins, max(len(offs) - 1, 0), dtype,
                      offs.ctypes.data_as(C.POINTER(C.c_int32)),
                      eb.ctypes.data_as(C.POINTER(C.c_int32)), renorm_topk, attn_max_heads,
                      int(gate), _p(score_bias), int(mi_topk_mask))
    h = C.c_void_p()
    code = _lib.smoes_plan_create(C.byref(desc), C.byref(h))
    return code, h


def smoes_plan_set_wait_limit(plan, limit_ns: int) -> int:
    return _lib.smoes_plan_set_wait_limit(plan, int(limit_ns))


def smoes_call_launches(plan, call: int) -> int:
    """Kernel launches one call makes on this plan (host query)."""
    return _lib.smoes_call_launches(plan, int(call))


def smoes_plan_destroy(plan):
    _lib.smoes_plan_destroy(plan)


def smoes_workspace_bytes(plan) -> int:
    return int(_lib.smoes_workspace_bytes(plan))


def smoes_workspace_init(plan, ws: torch.Tensor, stream=None) -> int:
    return _lib.smoes_workspace_init(plan, _p(ws), ws.numel() * ws.element_size(), _stream(stream))


def smoes_read_device_status(plan, ws: torch.Tensor, stream=None):
    n = C.c_int32(0)
    code = _lib.smoes_read_device_status(plan, _p(ws), _stream(stream), C.byref(n))
    return code, int(n.value)


def smoes_modality_score(plan, mode, M, ws, X=None, mu=None, var=None, tau=0.0, attn=None,
                         gmm=None, stream=None) -> int:
    """attn: dict with Q, K, B, H, S, hd, is_vision | m_prev, key_bias, sm_scale, causal,
    xattn_norm, x_norm (tensors or scalars)."""
    args = ScoreArgs()
    args.gauss = GaussArgs(_p(X), _p(mu), _p(var), float(tau))
    if attn is not None:
        a = attn
        args.attn = AttnArgs(_p(a["Q"]), _p(a["K"]), a["B"], a["H"], a["S"], a["hd"],
                             _p(a.get("is_vision")), _p(a.get("m_prev")), _p(a.get("key_bias")),
                             float(a["sm_scale"]), int(a.get("causal", 1)),
                             _p(a.get("xattn_norm")), _p(a.get("x_norm")))
    if gmm is not None:
        args.gmm = GmmArgs(_p(gmm["X"]), int(gmm["n_components"]), _p(gmm["log_pi"]), _p(gmm["mu"]),
                           _p(gmm["var"]), float(gmm.get("tau", 0.0)))
    return _lib.smoes_modality_score(plan, mode, C.byref(args), _p(M), _p(ws),
                                     ws.numel() * ws.element_size(), _stream(stream))


def smoes_router_fwd(plan, X, W, M_in, gauss, M_out, topk_idx, topk_w, bin_prob, joint, mi, loss,
                     ws, stream=None) -> int:
    """gauss: None (M_in given) or dict(mu=..., var=..., tau=...)."""
    g = None
    if gauss is not None:
        g = GaussArgs(None, _p(gauss["mu"]), _p(gauss["var"]), float(gauss.get("tau", 0.0)))
    return _lib.smoes_router_fwd(plan, _p(X), _p(W), _p(M_in), None if g is None else C.byref(g),
                                 _p(M_out), _p(topk_idx), _p(topk_w), _p(bin_prob), _p(joint),
                                 _p(mi), _p(loss), _p(ws), ws.numel() * ws.element_size(),
                                 _stream(stream))


def smoes_router_fwd_permute(plan, X, W, M_in, gauss, M_out, topk_idx, topk_w, bin_prob, joint, mi,
                             loss, home, is_vision, bin_offsets, perm_token, perm_mask, dispatch,
                             expert_counts, ws, stream=None) -> int:
    """smoes_router_fwd and smoes_bin_permute of its top-k in one call (one launch on bf16)."""
    g = None
    if gauss is not None:
        g = GaussArgs(None, _p(gauss["mu"]), _p(gauss["var"]), float(gauss.get("tau", 0.0)))
    return _lib.smoes_router_fwd_permute(plan, _p(X), _p(W), _p(M_in),
                                         None if g is None else C.byref(g), _p(M_out),
                                         _p(topk_idx), _p(topk_w), _p(bin_prob), _p(joint),
                                         _p(mi), _p(loss), _p(home), _p(is_vision),
                                         _p(bin_offsets), _p(perm_token), _p(perm_mask),
                                         _p(dispatch), _p(expert_counts), _p(ws),
                                         ws.numel() * ws.element_size(), _stream(stream))


def smoes_router_bwd(plan, X, W, M, topk_idx, d_topk_w, loss_scale, dW, accumulate_dW, dX,
                     dlogits, ws, stream=None) -> int:
    return _lib.smoes_router_bwd(plan, _p(X), _p(W), _p(M), _p(topk_idx), _p(d_topk_w),
                                 float(loss_scale), _p(dW), int(accumulate_dW), _p(dX),
                                 _p(dlogits), _p(ws), ws.numel() * ws.element_size(),
                                 _stream(stream))


def smoes_bin_permute(plan, topk_idx, home, is_vision, bin_offsets, perm_token, perm_mask,
                      dispatch, expert_counts, ws, stream=None) -> int:
    return _lib.smoes_bin_permute(plan, _p(topk_idx), _p(home), _p(is_vision), _p(bin_offsets),
                                  _p(perm_token), _p(perm_mask), _p(dispatch), _p(expert_counts),
                                  _p(ws), ws.numel() * ws.element_size(), _stream(stream))


def smoes_bin_permute_noalloc(plan, topk_idx, home, is_vision, bin_offsets, perm_token, perm_mask,
                              dispatch, expert_counts, stream=None) -> int:
    """The permutation without a workspace (scratch inside the library), for callers that cannot
    allocate device memory; see include/smoes.h for its limits and sharing rules."""
    return _lib.smoes_bin_permute_noalloc(plan, _p(topk_idx), _p(home), _p(is_vision),
                                          _p(bin_offsets), _p(perm_token), _p(perm_mask),
                                          _p(dispatch), _p(expert_counts), _stream(stream))


def smoes_gaussian_stats_update(plan, X, is_vision, beta, N, S_mu, S_var, mu, var, ws,
                                stream=None) -> int:
    return _lib.smoes_gaussian_stats_update(plan, _p(X), _p(is_vision), float(beta), _p(N), _p(S_mu),
                                            _p(S_var), _p(mu), _p(var), _p(ws),
                                            ws.numel() * ws.element_size(), _stream(stream))


def _attn_args(a):
    return AttnArgs(_p(a["Q"]), _p(a["K"]), a["B"], a["H"], a["S"], a["hd"], _p(a.get("is_vision")),
                    _p(a.get("m_prev")), _p(a.get("key_bias")), float(a["sm_scale"]),
                    int(a.get("causal", 1)), _p(a.get("xattn_norm")), _p(a.get("x_norm")))


def smoes_attention_fwd(plan, attn, V, n_kv_heads, O, M, ws, stream=None) -> int:
    """Attention forward with the vision score (O and M); attn as for smoes_modality_score."""
    args = _attn_args(attn)
    return _lib.smoes_attention_fwd(plan, C.byref(args), _p(V), int(n_kv_heads), _p(O), _p(M), _p(ws),
                                    ws.numel() * ws.element_size(), _stream(stream))


def smoes_bin_balance(plan, topk_idx, loss_scale, loss_bal, ws, f_e=None, P_e=None, stream=None) -> int:
    return _lib.smoes_bin_balance(plan, _p(topk_idx), float(loss_scale), _p(loss_bal), _p(f_e),
                                  _p(P_e), _p(ws), ws.numel() * ws.element_size(), _stream(stream))


def smoes_adaptive_bins(plan, expert_counts, beta, C_bar, expert_bin, f_spec=None, stream=None) -> int:
    return _lib.smoes_adaptive_bins(plan, _p(expert_counts), float(beta), _p(C_bar), _p(expert_bin),
                                    _p(f_spec), _stream(stream))


# ----------------------------------------------------------------------------- convenience

class Router:
    """Owns one plan and its workspace (torch-allocated) and the output buffers of one layer.

    Pure plumbing around the C calls above: allocation with torch, status checks, and the
    fwd -> bwd -> permute sequence.
    """

    def __init__(self, T, d, E, k, n_bins, sample_offsets, expert_bin, dtype=SMOES_BF16,
                 renorm_topk=0, attn_max_heads=0, device="cuda", gate=0, score_bias=None,
                 mi_topk_mask=0):
        code, self.plan = smoes_plan_create(T, d, E, k, n_bins, sample_offsets, expert_bin, dtype,
                                            renorm_topk, attn_max_heads, gate, score_bias,
                                            mi_topk_mask)
        _check(code, "smoes_plan_create")
        self.T, self.d, self.E, self.k, self.K = T, d, E, k, n_bins
        self.B = len(sample_offsets) - 1
        self.device = device
        nbytes = smoes_workspace_bytes(self.plan)
        self.ws = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=device)
        _check(smoes_workspace_init(self.plan, self.ws), "smoes_workspace_init")
        dev = device
        self.topk_idx = torch.empty((T, k), dtype=torch.int32, device=dev)
        self.topk_w = torch.empty((T, k), dtype=torch.float32, device=dev)
        self.bin_prob = torch.empty((T, n_bins), dtype=torch.float32, device=dev)
        self.joint = torch.empty((max(self.B, 1), 2, n_bins), dtype=torch.float32, device=dev)
        self.mi = torch.empty(max(self.B, 1), dtype=torch.float32, device=dev)
        self.loss = torch.empty(1, dtype=torch.float32, device=dev)
        self.M = torch.empty((T, 2), dtype=torch.float32, device=dev)
        cap = T * min(k, n_bins)
        self.bin_offsets = torch.empty(n_bins + 1, dtype=torch.int32, device=dev)
        self.perm_token = torch.empty(max(cap, 1), dtype=torch.int32, device=dev)
        self.perm_mask = torch.empty(max(cap, 1), dtype=torch.int32, device=dev)
        self.dispatch = torch.empty((n_bins, n_bins), dtype=torch.int32, device=dev)
        self.expert_counts = torch.empty((2, E), dtype=torch.int32, device=dev)

    def __del__(self):
        try:
            smoes_plan_destroy(self.plan)
        except Exception:
            pass

    def forward(self, X, W, M_in=None, mu=None, var=None, tau=0.0, bin_prob=True, stream=None):
        gauss = None if M_in is not None else dict(mu=mu, var=var, tau=tau)
        code = smoes_router_fwd(self.plan, X, W, M_in, gauss, None if M_in is not None else self.M,
                                self.topk_idx, self.topk_w, self.bin_prob if bin_prob else None,
                                self.joint, self.mi, self.loss, self.ws, stream)
        _check(code, "smoes_router_fwd")

    def forward_permute(self, X, W, M_in=None, mu=None, var=None, tau=0.0, bin_prob=True,
                        is_vision=None, home=None, stream=None):
        """forward() then permute() of its top-k, fused into one launch on bf16 plans."""
        gauss = None if M_in is not None else dict(mu=mu, var=var, tau=tau)
        code = smoes_router_fwd_permute(
            self.plan, X, W, M_in, gauss, None if M_in is not None else self.M, self.topk_idx,
            self.topk_w, self.bin_prob if bin_prob else None, self.joint, self.mi, self.loss, home,
            is_vision, self.bin_offsets, self.perm_token, self.perm_mask, self.dispatch,
            self.expert_counts if is_vision is not None else None, self.ws, stream)
        _check(code, "smoes_router_fwd_permute")

    def backward(self, X, W, M, dW, dX=None, dlogits=None, loss_scale=1.0, d_topk_w=None,
                 accumulate=False, stream=None):
        code = smoes_router_bwd(self.plan, X, W, M, self.topk_idx, d_topk_w, loss_scale, dW,
                                accumulate, dX, dlogits, self.ws, stream)
        _check(code, "smoes_router_bwd")

    def permute(self, is_vision=None, home=None, topk_idx=None, stream=None):
        code = smoes_bin_permute(self.plan, self.topk_idx if topk_idx is None else topk_idx, home,
                                 is_vision, self.bin_offsets, self.perm_token, self.perm_mask,
                                 self.dispatch, self.expert_counts if is_vision is not None else None,
                                 self.ws, stream)
        _check(code, "smoes_bin_permute")

    def modality_score(self, mode, M, **kw):
        code = smoes_modality_score(self.plan, mode, M, self.ws, **kw)
        _check(code, "smoes_modality_score")

    def device_status(self, stream=None):
        code, n_absent = smoes_read_device_status(self.plan, self.ws, stream)
        return code, n_absent
