"""Helpers for GPU-vs-oracle parity tests: run one router layer through the C ABI, run the fp64
oracle on the same inputs, and compare with the tolerances the build commits to:

  * integer outputs (top-k indices, permutation, dispatch, counts): bit-exact; top-k is compared
    on tokens whose oracle top-(k+1) logits have no adjacent gap below 1e-3 (near ties can
    legitimately order differently at fp32 accumulation); the excluded count is returned;
  * tensors: ||gpu - ref||_2 <= 2e-3 ||ref||_2 and max|gpu - ref| <= 2e-3 max|ref|;
  * scalars (MI per sample, loss): |gpu - ref| <= 2e-3 |ref| + 1e-9 nats;
  * outputs stored in bf16 (dX of a bf16 layer): the storage format alone has unit roundoff
    2^-8 (3.9e-3), above the 2e-3 bar, so each element must lie within one bf16 ulp of the exact
    oracle value (the correctly rounded value, or its neighbour when the fp32 result sits near a
    rounding boundary) plus 1e-4 max|ref| for the fp32 accumulation of elements that cancel to
    near zero, and the norm bar is 2e-3 + 2^-8. dX of a bf16 layer is formed from bf16 operands
    (dz rounded to bf16, fp32 accumulation: bf16 inputs, fp32 accumulate), so its elements also
    carry the rounding of dz to bf16, at most its unit roundoff 2^-8 times |dz_je| per term: the
    allowance adds 2^-8 sum_e |dz_je| |W_ed| (dx_operand_bound).
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import smoes_oracle as O

REL = 2e-3
ABS_NATS = 1e-9
TIE_GAP = 1e-3


def rel_err(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    nb = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / nb) if nb > 0 else float(np.linalg.norm(a))


def assert_tensor_close(gpu, ref, what, rel=REL):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    assert gpu.shape == ref.shape, (what, gpu.shape, ref.shape)
    assert np.all(np.isfinite(gpu)), f"{what}: non-finite values"
    scale = np.abs(ref).max() if ref.size else 0.0
    r = rel_err(gpu, ref)
    m = float(np.abs(gpu - ref).max()) if ref.size else 0.0
    assert r <= rel or (scale == 0 and m == 0), f"{what}: rel L2 error {r:.3e} > {rel}"
    assert m <= rel * scale or scale == 0, f"{what}: max abs error {m:.3e} > {rel} * {scale:.3e}"
    return r


def assert_scalar_close(gpu, ref, what):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    bad = np.abs(gpu - ref) > REL * np.abs(ref) + ABS_NATS
    assert not np.any(bad), f"{what}: {gpu[bad][:5]} vs {ref[bad][:5]}"


def bf16_ulp(x):
    """Spacing of bf16 numbers at |x| (8 significant bits)."""
    a = np.abs(np.asarray(x, np.float64))
    e = np.floor(np.log2(np.where(a > 0, a, 1e-38)))
    return np.where(a > 0, np.exp2(e - 7), 2.0 ** -133)


def dx_operand_bound(dz, W):
    """Largest effect on dX = dz W of rounding dz to bf16 (unit roundoff 2^-8 per element)."""
    return 2.0 ** -8 * (np.abs(np.asarray(dz, np.float64)) @ np.abs(np.asarray(W, np.float64)))


def assert_bf16_close(gpu, ref, what, operand_bound=None):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    assert np.all(np.isfinite(gpu)), f"{what}: non-finite values"
    err = np.abs(gpu - ref)
    floor = 1e-4 * (np.abs(ref).max() if ref.size else 0.0)
    if operand_bound is not None:
        floor = floor + operand_bound
    bad = err > bf16_ulp(ref) + floor
    assert not np.any(bad), (f"{what}: {int(bad.sum())} elements beyond one bf16 ulp; worst "
                             f"err {err[bad].max():.3e} at |ref| {np.abs(ref[bad]).max():.3e}")
    r = rel_err(gpu, ref)
    assert r <= REL + 2.0 ** -8, f"{what}: rel L2 error {r:.3e}"
    return r


def tie_free_tokens(z, k):
    """Tokens whose top-(k+1) logits (fp64 oracle) have all adjacent gaps >= TIE_GAP."""
    kk = min(k + 1, z.shape[1])
    top = -np.sort(-z, axis=1)[:, :kk]
    if kk < 2:
        return np.ones(z.shape[0], bool)
    return np.all(top[:, :-1] - top[:, 1:] >= TIE_GAP, axis=1)


def assert_valid_topk(idx, z, k):
    """For near-tie tokens: the chosen experts are distinct, each is a top-k choice within the
    tie gap, and they are listed in descending logit order within the tie gap."""
    if idx.shape[0] == 0:
        return
    assert np.all(np.sort(idx, axis=1)[:, 1:] != np.sort(idx, axis=1)[:, :-1]), "repeated expert"
    kth = -np.sort(-z, axis=1)[:, k - 1]
    chosen = np.take_along_axis(z, idx.astype(np.int64), axis=1)
    assert np.all(chosen >= kth[:, None] - TIE_GAP), "an expert outside the top-k was chosen"
    assert np.all(chosen[:, :-1] >= chosen[:, 1:] - TIE_GAP), "top-k not in descending order"


def to_dev(wl, dev):
    return wl.X.to(dev), wl.W.to(dev), wl.mu.to(dev), wl.var.to(dev)


def run_gpu(wl, bd, mode="gauss", M_in=None, d_topk_w=None, loss_scale=1.0, want_dx=True,
            want_dlogits=True, home=None, dev="cuda", fused=False):
    """One forward + backward + permutation through the C ABI; returns numpy outputs.
    fused: the permutation is requested from the forward call (smoes_router_fwd_permute)."""
    dtype = bd.SMOES_BF16 if wl.dtype == torch.bfloat16 else bd.SMOES_F32
    r = bd.Router(wl.T, wl.d, wl.E, wl.k, wl.n_bins, wl.sample_offsets, wl.expert_bin, dtype,
                  renorm_topk=wl.renorm_topk)
    X, W, mu, var = to_dev(wl, dev)
    hv = None if home is None else torch.as_tensor(home, dtype=torch.int32).to(dev)
    isv = torch.from_numpy(wl.is_vision).to(dev)
    fwd = (lambda **kw: r.forward_permute(is_vision=isv, home=hv, **kw)) if fused else r.forward
    if mode == "gauss":
        fwd(X=X, W=W, mu=mu, var=var, tau=wl.tau)
        M = r.M
    else:
        M = torch.as_tensor(M_in, dtype=torch.float32).to(dev).contiguous()
        fwd(X=X, W=W, M_in=M)
    dW = torch.full((wl.E, wl.d), float("nan"), dtype=torch.float32, device=dev)
    dX = torch.empty_like(X) if want_dx else None
    dl = torch.empty((wl.T, wl.E), dtype=torch.float32, device=dev) if want_dlogits else None
    dtw = None if d_topk_w is None else torch.as_tensor(d_topk_w, dtype=torch.float32).to(dev)
    r.backward(X, W, M, dW, dX=dX, dlogits=dl, loss_scale=loss_scale, d_topk_w=dtw)
    if not fused:
        r.permute(is_vision=isv, home=hv)
    code, n_absent = r.device_status()
    torch.cuda.synchronize()
    P = int(r.bin_offsets[-1].item())
    out = dict(status=code, n_absent=n_absent, M=M.cpu().numpy().astype(np.float64),
               topk_idx=r.topk_idx.cpu().numpy(), topk_w=r.topk_w.cpu().numpy(),
               bin_prob=r.bin_prob.cpu().numpy(), joint=r.joint.cpu().numpy(),
               mi=r.mi.cpu().numpy(), loss=float(r.loss.item()), dW=dW.cpu().numpy(),
               dX=None if dX is None else dX.float().cpu().numpy(),
               dlogits=None if dl is None else dl.cpu().numpy(),
               offsets=r.bin_offsets.cpu().numpy(), perm=r.perm_token[:P].cpu().numpy(),
               mask=r.perm_mask[:P].cpu().numpy().view(np.uint32),
               dispatch=r.dispatch.cpu().numpy(), expert_counts=r.expert_counts.cpu().numpy())
    del r
    return out


def run_oracle(wl, mode="gauss", M_in=None, loss_scale=1.0, d_topk_w=None, topk_idx_for_up=None):
    Xd = wl.X.double().numpy()
    Wd = wl.W.double().numpy()
    if mode == "gauss":
        M = O.gaussian_score(Xd, wl.mu.double().numpy(), wl.var.double().numpy(), wl.tau)
    else:
        M = np.asarray(M_in, np.float64)
    fwd = O.router_forward(Xd, Wd, M, wl.expert_bin, wl.n_bins, wl.sample_offsets, wl.k,
                           renorm=bool(wl.renorm_topk))
    N_B = wl.E // wl.n_bins
    dz = O.mi_grad_logits(M, fwd["g"], wl.expert_bin, wl.sample_offsets, fwd["tabs"], loss_scale, N_B)
    if d_topk_w is not None:
        dz = dz + O.topk_weight_grad_logits(fwd["g"], topk_idx_for_up, d_topk_w, bool(wl.renorm_topk))
    return dict(M=M, fwd=fwd, dz=dz, dW=dz.T @ Xd, dX=dz @ Wd)


def compare(wl, g, ref, check_dx=True, home=None):
    """Element-by-element comparison; returns a dict of measured errors and excluded counts."""
    res = {}
    fwd = ref["fwd"]
    assert g["status"] == 0, f"device status {g['status']}"
    res["M"] = assert_tensor_close(g["M"], ref["M"], "M")
    ok = tie_free_tokens(fwd["z"], wl.k)
    res["tie_excluded"] = int((~ok).sum())
    np.testing.assert_array_equal(g["topk_idx"][ok], fwd["topk_idx"][ok], err_msg="topk_idx")
    assert_valid_topk(g["topk_idx"][~ok], fwd["z"][~ok], wl.k)
    res["topk_w"] = assert_tensor_close(g["topk_w"][ok], fwd["topk_w"][ok], "topk_w")
    res["bin_prob"] = assert_tensor_close(g["bin_prob"], fwd["p"], "bin_prob")
    res["joint"] = assert_tensor_close(g["joint"][:wl.B], fwd["joint"], "joint")
    assert_scalar_close(g["mi"][:wl.B], fwd["mi"], "mi")
    assert_scalar_close(g["loss"], fwd["loss"], "loss")
    res["dlogits"] = assert_tensor_close(g["dlogits"], ref["dz"], "dlogits")
    res["dW"] = assert_tensor_close(g["dW"], ref["dW"], "dW")
    if check_dx and g["dX"] is not None:
        if wl.dtype == torch.bfloat16:
            res["dX"] = assert_bf16_close(g["dX"], ref["dX"], "dX",
                                          operand_bound=dx_operand_bound(ref["dz"], wl.W.double().numpy()))
        else:
            res["dX"] = assert_tensor_close(g["dX"], ref["dX"], "dX")
    # permutation, stage-wise: the oracle permutes the GPU's own top-k, bit for bit
    pr = O.bin_permute(g["topk_idx"], wl.expert_bin, wl.n_bins, home=home, is_vision=wl.is_vision)
    np.testing.assert_array_equal(g["offsets"], pr["offsets"], err_msg="bin_offsets")
    np.testing.assert_array_equal(g["perm"], pr["perm"], err_msg="perm_token")
    np.testing.assert_array_equal(g["mask"].astype(np.uint64), pr["mask"], err_msg="perm_mask")
    np.testing.assert_array_equal(g["dispatch"], pr["dispatch"], err_msg="dispatch")
    np.testing.assert_array_equal(g["expert_counts"], pr["expert_counts"], err_msg="expert_counts")
    return res
