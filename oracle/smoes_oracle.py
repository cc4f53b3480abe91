"""Plain fp64 CPU oracle of the SMoES modality-guided router (test infrastructure).

This module is TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import it. The product path (the CUDA library behind
``include/smoes.h`` and its Python binding) never calls it, and it shares no code, header,
table or helper with that path.

Every function follows the paper ("Soft Modality-Guided Expert Specialization in MoE-VLMs")
step by step, in float64, with numpy primitives (matmul, sort, log/exp) only. Where the paper
is silent the reading used is stated in the function's docstring.

Conventions
-----------
* Modality index m: 0 = vision, 1 = text (columns of the score matrix M [T, 2]).
* Samples are contiguous token ranges given by ``sample_offsets`` [B+1].
* ``expert_bin`` [E] maps each routed expert to its bin; every bin holds N_B = E / n_bins
  experts.
* Natural logarithms throughout.

Pins (what fixes this oracle independently of itself) live in ``tests/test_oracle_*.py``.
"""
from __future__ import annotations

import numpy as np

# A modality whose total soft mass in a sample is at or below this value is treated as absent
# from the sample (eq. 12 would be 0/0). Reading: its bin-averaged gating scores are 0.
MASS_EPS = 1e-12


def _f64(a):
    return np.asarray(a, dtype=np.float64)


# --------------------------------------------------------------------------------------------
# Soft modality scores (Sec. 3.2)
# --------------------------------------------------------------------------------------------

def gaussian_log_likelihood(X, mu, var):
    """Diagonal-Gaussian log-likelihood of every token under each modality, eq. (8).

    LL[j, m] = -1/2 * sum_d ( log var[m, d] + (x[j, d] - mu[m, d])^2 / var[m, d] ).

    X [T, d]; mu, var [2, d] (row 0 vision, row 1 text) -> LL [T, 2].
    """
    X, mu, var = _f64(X), _f64(mu), _f64(var)
    T = X.shape[0]
    LL = np.empty((T, 2))
    for m in range(2):
        LL[:, m] = -0.5 * np.sum(np.log(var[m])[None, :] + (X - mu[m][None, :]) ** 2 / var[m][None, :],
                                 axis=1)
    return LL


def gaussian_score(X, mu, var, tau):
    """Gaussian-statistics soft modality score, eq. (9): softmax over modalities of LL / tau.

    Returns M [T, 2] with M[:, 0] = vision score and M[:, 1] = text score.
    The paper's default temperature is tau = 0.5 * D with D the hidden size (Sec. 4.1).
    """
    LL = gaussian_log_likelihood(X, mu, var) / float(tau)
    LL = LL - LL.max(axis=1, keepdims=True)
    e = np.exp(LL)
    return e / e.sum(axis=1, keepdims=True)


def gmm_log_likelihood(X, log_pi, mu, var):
    """Log-likelihood of every token under each modality's diagonal Gaussian mixture: the
    estimator the paper explores beyond the single Gaussian of eq. (8) (supplementary, "GMM
    estimator" with k components).

    LL[j, m] = log sum_c pi[m, c] N(x_j; mu[m, c], diag var[m, c])
             = logsumexp_c ( log pi[m, c] - 1/2 sum_d ( log(2 pi) + log var[m, c, d]
                                                       + (x_jd - mu[m, c, d])^2 / var[m, c, d] ) ).
    The log(2 pi) term is the same for both modalities and is kept so that the values are true
    log-densities (it cancels in the score).

    X [T, d]; log_pi [2, C]; mu, var [2, C, d] -> LL [T, 2].
    """
    X, log_pi, mu, var = _f64(X), _f64(log_pi), _f64(mu), _f64(var)
    T, d = X.shape
    C = mu.shape[1]
    LL = np.empty((T, 2))
    for m in range(2):
        q = np.empty((T, C))
        for c in range(C):
            q[:, c] = log_pi[m, c] - 0.5 * np.sum(np.log(2.0 * np.pi) + np.log(var[m, c])[None, :]
                                                  + (X - mu[m, c][None, :]) ** 2 / var[m, c][None, :],
                                                  axis=1)
        top = q.max(axis=1, keepdims=True)
        LL[:, m] = top[:, 0] + np.log(np.sum(np.exp(q - top), axis=1))
    return LL


def gmm_score(X, log_pi, mu, var, tau):
    """Soft modality score with the GMM estimator: eq. (9) applied to the mixture
    log-likelihoods of gmm_log_likelihood (C = 1 gives the Gaussian score of eqs. 8-9)."""
    LL = gmm_log_likelihood(X, log_pi, mu, var) / float(tau)
    LL = LL - LL.max(axis=1, keepdims=True)
    e = np.exp(LL)
    return e / e.sum(axis=1, keepdims=True)


def attention_vision_mass(Q, K, m_keys, sm_scale, causal=True, key_bias=None, queries=None):
    """Attention-accumulated vision score, eqs. (2)-(3).

    For sequence b and query j the aggregated score is
        Mtilde_v[b, j] = (1/H) * sum_h sum_{j'} Attn_h[j, j'] * m[b, j'],
    where Attn_h is the row-softmax of sm_scale * q_{b,h,j} . k_{b,h,j'} (+ key_bias[b, j'])
    over the keys j' <= j when causal, i.e. the attention matrix averaged over heads (eq. 3)
    applied to the previous layer's vision score m (eq. 2 gives the hard labels at layer 0).

    Q, K [B, H, S, hd]; m_keys [B, S]; key_bias [B, S] or None.
    queries: None for all (b, j), else an int array [n, 2] of (b, j) rows to evaluate.
    Returns Mtilde_v as [B, S] (queries None) or [n].
    """
    Q, K, m_keys = _f64(Q), _f64(K), _f64(m_keys)
    B, H, S, _ = Q.shape
    bias = np.zeros((B, S)) if key_bias is None else _f64(key_bias)

    def one_query(b, j):
        n = j + 1 if causal else S
        logits = sm_scale * np.einsum('hd,hsd->hs', Q[b, :, j, :], K[b, :, :n, :]) + bias[b, None, :n]
        logits = logits - logits.max(axis=1, keepdims=True)
        w = np.exp(logits)
        w = w / w.sum(axis=1, keepdims=True)
        return float(np.mean(w @ m_keys[b, :n]))

    if queries is None:
        out = np.empty((B, S))
        for b in range(B):
            for h_block in range(0, S, 256):
                # blocked evaluation of all queries of one sequence (same arithmetic as one_query)
                j0, j1 = h_block, min(S, h_block + 256)
                n = j1 if causal else S
                logits = sm_scale * np.einsum('hqd,hsd->hqs', Q[b, :, j0:j1, :], K[b, :, :n, :])
                logits = logits + bias[b, None, None, :n]
                if causal:
                    jj = np.arange(j0, j1)[:, None]
                    kk = np.arange(n)[None, :]
                    logits = np.where((kk <= jj)[None, :, :], logits, -np.inf)
                logits = logits - logits.max(axis=2, keepdims=True)
                w = np.exp(logits)
                w = w / w.sum(axis=2, keepdims=True)
                out[b, j0:j1] = np.mean(w @ m_keys[b, :n], axis=0)
        return out
    queries = np.asarray(queries)
    return np.array([one_query(int(b), int(j)) for b, j in queries])


def attention_forward_with_mass(Q, K, V, m_keys, sm_scale, causal=True, key_bias=None):
    """Causal attention output and the aggregated vision score in one pass, the fused form of
    eqs. (2)-(3): the score is attention with the carried score m as one more value column, so
    O_ext = Attn [V | m] gives the layer's output (first dv columns) and, averaged over heads, its
    last column is Mtilde_v. Grouped-query attention: K and V may have Hkv = H / G heads; query
    head h reads key/value head h // G.

    Q [B, H, S, hd]; K [B, Hkv, S, hd]; V [B, Hkv, S, dv]; m_keys [B, S]; key_bias [B, S] or None.
    Returns (O [B, H, S, dv], Mtilde_v [B, S]).
    """
    Q, K, V, m_keys = _f64(Q), _f64(K), _f64(V), _f64(m_keys)
    B, H, S, _ = Q.shape
    Hkv = K.shape[1]
    G = H // Hkv
    bias = np.zeros((B, S)) if key_bias is None else _f64(key_bias)
    O = np.empty((B, H, S, V.shape[3]))
    mass = np.zeros((B, S))
    for b in range(B):
        for h in range(H):
            hk = h // G
            logits = sm_scale * (Q[b, h] @ K[b, hk].T) + bias[b][None, :]
            if causal:
                logits = np.where(np.tri(S, dtype=bool), logits, -np.inf)
            logits = logits - logits.max(axis=1, keepdims=True)
            w = np.exp(logits)
            w = w / w.sum(axis=1, keepdims=True)
            ext = w @ np.concatenate([V[b, hk], m_keys[b][:, None]], axis=1)
            O[b, h] = ext[:, :-1]
            mass[b] += ext[:, -1] / H
    return O, mass


def residual_score_update(M_tilde, M_prev, xattn_norm, x_norm):
    """Residual-weighted score update, eq. (4):
    M_next = (|x_attn| * Mtilde + |x| * M_prev) / (|x_attn| + |x|), per token and modality.
    """
    a = _f64(xattn_norm)
    r = _f64(x_norm)
    return (a * _f64(M_tilde) + r * _f64(M_prev)) / (a + r)


# --------------------------------------------------------------------------------------------
# Router: gate, softmax, top-k, bins (Sec. 3.1, Sec. 3.3)
# --------------------------------------------------------------------------------------------

def gate_logits(X, W):
    """Gate logits z = W_gate x for every token (Sec. 3.1); X [T, d], W [E, d] -> z [T, E]."""
    return _f64(X) @ _f64(W).T


def softmax_gate(z):
    """Gating scores g = softmax(z) over the routed experts (Sec. 3.1)."""
    z = _f64(z)
    e = np.exp(z - z.max(axis=1, keepdims=True))
    return e / e.sum(axis=1, keepdims=True)


def topk_route(z, g, k, renorm=False):
    """Top-k expert choice (Sec. 3.1).

    Order: descending logit; equal logits are ordered by ascending expert index (reading: the
    paper does not fix a tie rule). Weights are the softmax scores of the chosen experts, or
    those scores renormalised over the top-k when ``renorm``.
    Returns (idx int32 [T, k], w float64 [T, k]).
    """
    z = _f64(z)
    order = np.argsort(-z, axis=1, kind='stable')[:, :k]
    w = np.take_along_axis(_f64(g), order, axis=1)
    if renorm:
        w = w / w.sum(axis=1, keepdims=True)
    return order.astype(np.int32), w


def sigmoid_gate(z, score_bias=None, k=None):
    """Sigmoid router with a selection bias (the router of Moonlight-MoE in the paper's backbone
    table): affinities s = sigmoid(z); experts chosen by the top-k of s + b (the bias only steers
    the choice); top-k weights s / sum of the chosen s. Readings: the gating scores g that enter
    eq. (12) (and the bin sums) are the affinities normalised over all experts, g = s / sum_e s,
    so that p_j. is a distribution as with the softmax router; ties in s + b go to the lower
    expert index.

    z [T, E]; score_bias [E] or None. Returns dict(s, g, topk_idx [T, k] int32, topk_w [T, k]).
    """
    z = _f64(z)
    s = 1.0 / (1.0 + np.exp(-z))
    g = s / s.sum(axis=1, keepdims=True)
    out = dict(s=s, g=g)
    if k is not None:
        key = s + (0.0 if score_bias is None else _f64(score_bias)[None, :])
        idx = np.argsort(-key, axis=1, kind='stable')[:, :k]
        w = np.take_along_axis(s, idx, axis=1)
        out.update(topk_idx=idx.astype(np.int32), topk_w=w / w.sum(axis=1, keepdims=True))
    return out


def sigmoid_grad_logits(s, dL_dg):
    """Gradient at the logits of a loss given through g = s / sum s, s = sigmoid(z):
    dL/dz_e = s_e (1 - s_e) (dL/dg_e - sum_e' g_e' dL/dg_e') / sum s."""
    s, dL_dg = _f64(s), _f64(dL_dg)
    S = s.sum(axis=1, keepdims=True)
    g = s / S
    return s * (1.0 - s) * (dL_dg - np.sum(g * dL_dg, axis=1, keepdims=True)) / S


def topk_masked_gate(g, topk_idx):
    """The top-k-masked reading of g in eq. (12): the gate restricted to the chosen experts and
    renormalised over them (zero elsewhere), so that its bin sums still form a distribution."""
    g = _f64(g)
    out = np.zeros_like(g)
    idx = np.asarray(topk_idx, dtype=np.int64)
    sel = np.take_along_axis(g, idx, axis=1)
    np.put_along_axis(out, idx, sel / sel.sum(axis=1, keepdims=True), axis=1)
    return out


def bin_probs(g, expert_bin, n_bins):
    """Per-bin routing probability p[j, k] = sum_{e in B_k} g[j, e] (the inner sum of eq. 12)."""
    g = _f64(g)
    expert_bin = np.asarray(expert_bin)
    p = np.zeros((g.shape[0], n_bins))
    for kb in range(n_bins):
        p[:, kb] = g[:, expert_bin == kb].sum(axis=1)
    return p


# --------------------------------------------------------------------------------------------
# Inter-bin mutual information (Sec. 3.4)
# --------------------------------------------------------------------------------------------

def sample_joint(M, p, N_B):
    """Joint table of one sample, eqs. (12)-(14).

    M [n, 2] soft scores, p [n, K] bin probabilities of the sample's tokens.
      A[m]      = sum_j M[j, m]
      Sbar[m,k] = sum_j M[j, m] p[j, k] / (N_B * A[m])           (12)
      P[m,k]    = Sbar[m,k] / sum Sbar                            (13)
      I         = sum_{m,k} P log(P / (P_m P_k)),  0 log 0 = 0    (14)
    A modality with A[m] <= MASS_EPS is absent: its Sbar row is 0 (reading of 0/0).
    Returns dict with A, N, Sbar, Z, P, Pm, Pk, I.
    """
    M, p = _f64(M), _f64(p)
    K = p.shape[1]
    A = M.sum(axis=0)
    N = M.T @ p
    Sbar = np.zeros((2, K))
    for m in range(2):
        if A[m] > MASS_EPS:
            Sbar[m] = N[m] / (N_B * A[m])
    Z = Sbar.sum()
    P = Sbar / Z
    Pm = P.sum(axis=1)
    Pk = P.sum(axis=0)
    I = 0.0
    for m in range(2):
        for kb in range(K):
            if P[m, kb] > 0.0:
                I += P[m, kb] * np.log(P[m, kb] / (Pm[m] * Pk[kb]))
    return dict(A=A, N=N, Sbar=Sbar, Z=Z, P=P, Pm=Pm, Pk=Pk, I=I)


def mi_loss(M, p, sample_offsets, N_B):
    """Per-sample MI (eq. 14) and the MI loss of one layer, eq. (15): L = -(1/B) sum_i I_i.

    M [T, 2], p [T, K], sample_offsets [B+1], N_B experts per bin.
    Returns (mi [B], joint P [B, 2, K], loss, per-sample tables).
    """
    offs = np.asarray(sample_offsets)
    B = len(offs) - 1
    K = p.shape[1]
    mis = np.zeros(B)
    joint = np.zeros((B, 2, K))
    tabs = []
    for i in range(B):
        s, e = int(offs[i]), int(offs[i + 1])
        tab = sample_joint(M[s:e], p[s:e], N_B)
        mis[i] = tab['I']
        joint[i] = tab['P']
        tabs.append(tab)
    loss = -mis.sum() / B if B > 0 else 0.0
    return mis, joint, loss, tabs


def mi_grad_logits(M, g, expert_bin, sample_offsets, tabs, loss_scale, N_B):
    """Gradient of loss_scale * L_MI with respect to the gate logits.

    Derivation from eqs. (12)-(15), with the soft scores M (hence A) held constant
    (stop-gradient; reading: the scores are guide signals, not functions of the gate):
      dI/dSbar[m,k] = (log(P[m,k] / (P_m P_k)) - I) / Z
      u[j,k]        = sum_m M[j,m] * dI/dSbar[m,k] / (N_B A[m])        (= dI/dg[j,e], e in B_k)
      dI/dz[j,e]    = g[j,e] * (u[j, bin(e)] - sum_e' g[j,e'] u[j, bin(e')])   (softmax Jacobian)
      dL/dz         = -(loss_scale / B) * dI/dz.
    Absent modalities (A[m] <= MASS_EPS) contribute nothing.
    """
    M, g = _f64(M), _f64(g)
    expert_bin = np.asarray(expert_bin)
    offs = np.asarray(sample_offsets)
    B = len(offs) - 1
    dz = np.zeros_like(g)
    for i in range(B):
        s, e = int(offs[i]), int(offs[i + 1])
        tab = tabs[i]
        K = tab['P'].shape[1]
        u_coef = np.zeros((2, K))
        for m in range(2):
            if tab['A'][m] > MASS_EPS:
                with np.errstate(divide='ignore', invalid='ignore'):
                    ratio = np.where(tab['P'][m] > 0, tab['P'][m] / (tab['Pm'][m] * tab['Pk']), 1.0)
                dI_dS = (np.log(ratio) - tab['I']) / tab['Z']
                u_coef[m] = dI_dS / (N_B * tab['A'][m])
        u = M[s:e] @ u_coef                       # [n, K]
        ue = u[:, expert_bin]                     # [n, E]
        gi = g[s:e]
        dI_dz = gi * (ue - np.sum(gi * ue, axis=1, keepdims=True))
        dz[s:e] = -(loss_scale / B) * dI_dz
    return dz


def topk_weight_grad_logits(g, topk_idx, d_topk_w, renorm=False):
    """Gradient reaching the gate logits from an upstream gradient of the top-k weights.

    The weights are w_i = g[e_i] (or g[e_i] / sum_i' g[e_i'] when renormalised); the chain rule
    through that renormalisation and through the softmax gives the returned dL/dz [T, E].
    """
    g = _f64(g)
    T, E = g.shape
    idx = np.asarray(topk_idx)
    d = _f64(d_topk_w)
    dg = np.zeros((T, E))
    if renorm:
        gsel = np.take_along_axis(g, idx, axis=1)
        Gs = gsel.sum(axis=1, keepdims=True)
        w = gsel / Gs
        dsel = (d - np.sum(d * w, axis=1, keepdims=True)) / Gs
    else:
        dsel = d
    rows = np.repeat(np.arange(T), idx.shape[1])
    np.add.at(dg, (rows, idx.reshape(-1)), dsel.reshape(-1))
    return g * (dg - np.sum(g * dg, axis=1, keepdims=True))


# --------------------------------------------------------------------------------------------
# Bin-grouped permutation and EP dispatch counts (Sec. 4.5, DeDup)
# --------------------------------------------------------------------------------------------

def expert_slots(expert_bin, n_bins):
    """Position of every expert inside its bin (experts of a bin in ascending index order)."""
    expert_bin = np.asarray(expert_bin)
    slot = np.zeros(len(expert_bin), dtype=np.int64)
    for kb in range(n_bins):
        members = np.nonzero(expert_bin == kb)[0]
        slot[members] = np.arange(len(members))
    return slot


def default_home(T, n_bins):
    """Device a token lives on before dispatch (reading): a contiguous split over n_bins devices,
    home(j) = floor(j * n_bins / T)."""
    j = np.arange(T, dtype=np.int64)
    return (j * n_bins) // max(T, 1)


def bin_permute(topk_idx, expert_bin, n_bins, home=None, is_vision=None):
    """De-duplicated bin dispatch (Sec. 4.5): one entry per unique (token, bin) pair.

    A token is sent once to a bin even if several of its top-k experts live there; the entry
    carries a bit mask of those experts (bit = the expert's slot inside the bin).
    Order: bin ascending, token ascending inside a bin.
    dispatch[h, k] counts unique pairs whose token lives on device h.
    expert_counts[m, e] counts the tokens of hard modality m that chose expert e (eq. 10's C).
    Returns dict(offsets [K+1], perm [P], mask [P], dispatch [K, K], expert_counts [2, E] or None).
    """
    idx = np.asarray(topk_idx, dtype=np.int64)
    T, k = idx.shape
    expert_bin = np.asarray(expert_bin, dtype=np.int64)
    E = len(expert_bin)
    K = n_bins
    slot = expert_slots(expert_bin, K)
    home = default_home(T, K) if home is None else np.asarray(home, dtype=np.int64)

    sel_mask = np.zeros((T, K), dtype=np.uint64)          # bit mask of chosen experts per bin
    bins = expert_bin[idx]                                # [T, k]
    bits = np.left_shift(np.uint64(1), slot[idx].astype(np.uint64))
    for c in range(k):
        np.bitwise_or.at(sel_mask, (np.arange(T), bins[:, c]), bits[:, c])
    present = sel_mask != 0                               # [T, K] unique pairs
    counts = present.sum(axis=0)
    offsets = np.zeros(K + 1, dtype=np.int64)
    offsets[1:] = np.cumsum(counts)
    # counting sort by bin, stable in token order
    perm_parts, mask_parts = [], []
    for kb in range(K):
        toks = np.nonzero(present[:, kb])[0]
        perm_parts.append(toks)
        mask_parts.append(sel_mask[toks, kb])
    perm = np.concatenate(perm_parts) if perm_parts else np.zeros(0, np.int64)
    mask = np.concatenate(mask_parts) if mask_parts else np.zeros(0, np.uint64)
    dispatch = np.zeros((K, K), dtype=np.int64)
    jj, kk = np.nonzero(present)
    np.add.at(dispatch, (home[jj], kk), 1)
    ec = None
    if is_vision is not None:
        lab = np.where(np.asarray(is_vision) != 0, 0, 1)
        ec = np.zeros((2, E), dtype=np.int64)
        np.add.at(ec, (np.repeat(lab, k), idx.reshape(-1)), 1)
    return dict(offsets=offsets, perm=perm, mask=mask, dispatch=dispatch, expert_counts=ec)


# --------------------------------------------------------------------------------------------
# Composite steps: one router layer forward and backward
# --------------------------------------------------------------------------------------------

def router_forward(X, W, M, expert_bin, n_bins, sample_offsets, k, renorm=False):
    """Forward of one MoE router layer with the inter-bin MI regulariser (Secs. 3.1, 3.4).

    X [T, d], W [E, d], M [T, 2] soft modality scores. Returns a dict with z, g, topk_idx,
    topk_w, p, mi [B], joint [B, 2, K], loss and the per-sample tables (for the backward).
    """
    expert_bin = np.asarray(expert_bin)
    N_B = len(expert_bin) // n_bins
    z = gate_logits(X, W)
    g = softmax_gate(z)
    idx, w = topk_route(z, g, k, renorm)
    p = bin_probs(g, expert_bin, n_bins)
    mis, joint, loss, tabs = mi_loss(_f64(M), p, sample_offsets, N_B)
    return dict(z=z, g=g, topk_idx=idx, topk_w=w, p=p, mi=mis, joint=joint, loss=loss, tabs=tabs)


def router_backward(X, W, M, fwd, expert_bin, sample_offsets, loss_scale, d_topk_w=None,
                    renorm=False):
    """Backward of loss_scale * L_MI (+ an optional upstream gradient of the top-k weights).

    dL/dz from mi_grad_logits (+ topk_weight_grad_logits), then dW = dz^T X and dX = dz W.
    Returns (dz [T, E], dW [E, d], dX [T, d]).
    """
    expert_bin = np.asarray(expert_bin)
    N_B = len(expert_bin) // fwd['p'].shape[1]
    dz = mi_grad_logits(M, fwd['g'], expert_bin, sample_offsets, fwd['tabs'], loss_scale, N_B)
    if d_topk_w is not None:
        dz = dz + topk_weight_grad_logits(fwd['g'], fwd['topk_idx'], d_topk_w, renorm)
    dW = dz.T @ _f64(X)
    dX = dz @ _f64(W)
    return dz, dW, dX


def mi_grad_gate(M, expert_bin, sample_offsets, tabs, loss_scale, N_B):
    """Gradient of loss_scale * L_MI with respect to the gate values that enter eq. (12) (the
    quantity summed into the bins): -(loss_scale / B) u[j, bin(e)], with u as in mi_grad_logits.
    Returns [T, E]."""
    M = _f64(M)
    expert_bin = np.asarray(expert_bin)
    offs = np.asarray(sample_offsets)
    B = len(offs) - 1
    out = np.zeros((M.shape[0], len(expert_bin)))
    for i in range(B):
        s, e = int(offs[i]), int(offs[i + 1])
        tab = tabs[i]
        K = tab['P'].shape[1]
        u_coef = np.zeros((2, K))
        for m in range(2):
            if tab['A'][m] > MASS_EPS:
                with np.errstate(divide='ignore', invalid='ignore'):
                    ratio = np.where(tab['P'][m] > 0, tab['P'][m] / (tab['Pm'][m] * tab['Pk']), 1.0)
                u_coef[m] = (np.log(ratio) - tab['I']) / tab['Z'] / (N_B * tab['A'][m])
        out[s:e] = -(loss_scale / B) * (M[s:e] @ u_coef)[:, expert_bin]
    return out


def softmax_grad_logits(g, dL_dg):
    """Chain rule through g = softmax(z): dL/dz = g (dL/dg - sum_e' g_e' dL/dg_e')."""
    g, dL_dg = _f64(g), _f64(dL_dg)
    return g * (dL_dg - np.sum(g * dL_dg, axis=1, keepdims=True))


def masked_gate_grad(g, topk_idx, dL_dgt):
    """Chain rule through the top-k-masked gate gt = g / sum_sel g on the chosen experts:
    dL/dg_e = (dL/dgt_e - sum_sel gt dL/dgt) / sum_sel g for chosen e, 0 elsewhere."""
    g, dL_dgt = _f64(g), _f64(dL_dgt)
    idx = np.asarray(topk_idx, dtype=np.int64)
    gs = np.take_along_axis(g, idx, axis=1)
    G = gs.sum(axis=1, keepdims=True)
    ds = np.take_along_axis(dL_dgt, idx, axis=1)
    out = np.zeros_like(g)
    np.put_along_axis(out, idx, (ds - np.sum(gs / G * ds, axis=1, keepdims=True)) / G, axis=1)
    return out


def router_forward_variant(X, W, M, expert_bin, n_bins, sample_offsets, k, gate='softmax',
                           score_bias=None, mask=False, renorm=False, topk_idx=None):
    """Forward of one router layer for the router variants of the backbone table and of the
    readings of eq. (12): gate 'softmax' (Sec. 3.1) or 'sigmoid' (sigmoid_gate, with an optional
    selection bias; its top-k weights are always renormalised), and the gate entering eq. (12)
    either dense (all experts) or top-k-masked (topk_masked_gate). Same outputs as
    router_forward plus 'gq', the gate values summed into the bins, and 's' (sigmoid only).
    topk_idx: a given choice instead of the gate's own (stage-wise comparisons of what follows
    the choice); the weights are then those of the given experts."""
    z = gate_logits(X, W)
    if gate == 'softmax':
        g = softmax_gate(z)
        idx, w = topk_route(z, g, k, renorm)
        s = None
    elif gate == 'sigmoid':
        out = sigmoid_gate(z, score_bias, k)
        g, idx, w, s = out['g'], out['topk_idx'], out['topk_w'], out['s']
    else:
        raise ValueError(gate)
    if topk_idx is not None:
        idx = np.asarray(topk_idx).astype(np.int32)
        src = g if gate == 'softmax' else s
        w = np.take_along_axis(src, idx.astype(np.int64), axis=1)
        if gate == 'sigmoid' or renorm:
            w = w / w.sum(axis=1, keepdims=True)
    gq = topk_masked_gate(g, idx) if mask else g
    N_B = len(expert_bin) // n_bins
    p = bin_probs(gq, expert_bin, n_bins)
    mis, joint, loss, tabs = mi_loss(_f64(M), p, sample_offsets, N_B)
    return dict(z=z, g=g, s=s, gq=gq, topk_idx=idx, topk_w=w, p=p, mi=mis, joint=joint, loss=loss,
                tabs=tabs, gate=gate, mask=mask)


def router_backward_variant(X, W, M, fwd, expert_bin, sample_offsets, loss_scale):
    """Backward of loss_scale * L_MI for router_forward_variant: dL/d(gate values of eq. 12)
    (mi_grad_gate), through the top-k mask when used (masked_gate_grad), then through the gate
    (softmax_grad_logits or sigmoid_grad_logits); dW = dz^T X, dX = dz W."""
    N_B = len(expert_bin) // fwd['p'].shape[1]
    dgq = mi_grad_gate(M, expert_bin, sample_offsets, fwd['tabs'], loss_scale, N_B)
    dg = masked_gate_grad(fwd['g'], fwd['topk_idx'], dgq) if fwd['mask'] else dgq
    dz = softmax_grad_logits(fwd['g'], dg) if fwd['gate'] == 'softmax' else sigmoid_grad_logits(fwd['s'], dg)
    return dz, dz.T @ _f64(X), dz @ _f64(W)


def msi(expert_counts):
    """Modality Specialization Index, eqs. (18)-(19), for one layer from counts C [2, E]
    (row 0 vision, row 1 text). Returns a value in [0, 1]."""
    C = _f64(expert_counts)
    share = C / C.sum(axis=1, keepdims=True)            # C_{m,e} / sum_e' C_{m,e'}
    Ct = share / share.sum(axis=0, keepdims=True)       # eq. (18)
    return float(np.mean(2.0 * np.abs(Ct[1] - 0.5)))    # eq. (19), text row


# --------------------------------------------------------------------------------------------
# Online statistics and momentum-adaptive binning (Secs. 3.2 and 3.3)
# --------------------------------------------------------------------------------------------

def gaussian_stats_empty(d):
    """The empty state (N, S_mu, S_var) of the per-modality statistics: all zeros."""
    return np.zeros(2), np.zeros((2, d)), np.zeros((2, d))


def gaussian_stats_update(state, X, is_vision, beta):
    """One step of the EMA variant of Welford's algorithm, eqs. (5)-(7), for both modalities.

    state = (N [2], S_mu [2, d], S_var [2, d]) at step t-1; X [T, d]; is_vision [T] (hard labels:
    T_m is the set of the batch's modality-m tokens); beta: the EMA decay. Returns the state at t:

        N_t     = beta N_{t-1} + |T_m|                                                  (5)
        S_mu,t  = beta S_mu,t-1 + |T_m| mu_{T_m}                                        (6)
        S_var,t = beta S_var,t-1 + sum_{x in T_m} (x - mu_{T_m})^2
                  + (mu_{T_m} - S_mu,t-1 / N_{t-1})^2 beta N_{t-1} |T_m| / (beta N_{t-1} + |T_m|)  (7)

    with mu_{T_m} the batch mean of modality m. Readings: the last term of (7) is zero when
    N_{t-1} = 0 (empty state: the factor is 0 and the previous mean undefined) or |T_m| = 0 (no
    token of the modality in the batch: the batch mean undefined, the factor 0).
    """
    N0, Smu0, Svar0 = (_f64(a) for a in state)
    X = _f64(X)
    lab = np.asarray(is_vision)
    N, Smu, Svar = np.empty(2), np.empty_like(Smu0), np.empty_like(Svar0)
    for m, rows in enumerate((lab == 1, lab == 0)):       # row 0 vision, row 1 text
        Xm = X[rows]
        n = Xm.shape[0]
        N[m] = beta * N0[m] + n
        if n == 0:
            Smu[m] = beta * Smu0[m]
            Svar[m] = beta * Svar0[m]
            continue
        mu_b = Xm.mean(axis=0)
        Smu[m] = beta * Smu0[m] + n * mu_b
        Svar[m] = beta * Svar0[m] + np.sum((Xm - mu_b[None, :]) ** 2, axis=0)
        if N0[m] > 0:
            w = beta * N0[m] * n / (beta * N0[m] + n)
            Svar[m] += (mu_b - Smu0[m] / N0[m]) ** 2 * w
    return N, Smu, Svar


def gaussian_stats(state):
    """The distribution parameters of Sec. 3.2: mu_m = S_mu / N and var_m = S_var / N, [2, d]."""
    N, Smu, Svar = (_f64(a) for a in state)
    return Smu / N[:, None], Svar / N[:, None]


def expert_load_ema(C_bar, C, beta):
    """Eq. (10): C_bar_t = beta C_bar_{t-1} + (1 - beta) C, per modality and expert [2, E]."""
    return beta * _f64(C_bar) + (1.0 - beta) * _f64(C)


def text_bias(C_bar):
    """Eq. (11): f_spec(e) = C_bar[text, e] / (C_bar[text, e] + C_bar[vision, e]), [E].

    Reading: an expert with no load from either modality (0/0) is neutral, f = 1/2.
    """
    C_bar = _f64(C_bar)
    tot = C_bar[0] + C_bar[1]
    return np.where(tot > 0, C_bar[1] / np.where(tot > 0, tot, 1.0), 0.5)


def adaptive_bins(f_spec, n_bins):
    """Momentum-adaptive binning (Sec. 3.3): experts sorted by f_spec and cut into n_bins runs of
    N_B = E / n_bins consecutive experts. Readings: ascending order (bin 0 holds the most
    vision-biased experts), equal scores kept in expert-index order. Returns expert_bin [E]."""
    f = _f64(f_spec)
    E = f.shape[0]
    order = np.argsort(f, kind="stable")
    expert_bin = np.empty(E, dtype=np.int32)
    expert_bin[order] = np.arange(E) // (E // n_bins)
    return expert_bin


# --------------------------------------------------------------------------------------------
# Bin-level load balance (Sec. 3.5)
# --------------------------------------------------------------------------------------------

def bin_balance_loss(g, topk_idx, expert_bin, n_bins):
    """Bin-level load-balance loss of one layer, eq. (16):
        L_bal = sum_k N_B sum_{e in B_k} f_e P_e,
    with f_e and P_e taken over the tokens routed to bin B_k. Readings (the paper defers to the
    load-balance terms of its preliminaries): U_k is the set of tokens with at least one of
    their top-k experts in B_k; f_e = (selections of e) / (selections of all experts of B_k),
    P_e = mean over j in U_k of g_je / sum_{e' in B_k} g_je' (the gate renormalised inside the
    bin). Both sum to 1 over a bin, so a bin whose load is spread evenly gives 1. A bin that no
    token selects contributes 0. With one bin this is the standard loss N_e sum_e f_e P_e of the
    preliminaries (f_e over all selections, P_e the mean gate).

    g [T, E] softmax scores, topk_idx [T, k] -> (L, dict(f [E], P [E], used [K] bool)).
    """
    g = _f64(g)
    T, E = g.shape
    eb = np.asarray(expert_bin)
    N_B = E // n_bins
    sel = np.zeros((T, E), dtype=bool)
    sel[np.arange(T)[:, None], np.asarray(topk_idx)] = True
    f = np.zeros(E)
    P = np.zeros(E)
    used = np.zeros(n_bins, dtype=bool)
    L = 0.0
    for k in range(n_bins):
        members = np.nonzero(eb == k)[0]
        U = sel[:, members].any(axis=1)                       # tokens routed to bin k
        n_sel = sel[:, members].sum()
        if n_sel == 0:
            continue
        used[k] = True
        f[members] = sel[:, members].sum(axis=0) / n_sel
        gk = g[U][:, members]
        P[members] = np.mean(gk / gk.sum(axis=1, keepdims=True), axis=0)
        L += N_B * float(np.sum(f[members] * P[members]))
    return L, dict(f=f, P=P, used=used)


def sigmoid_topk_weight_grad_logits(s, topk_idx, d_topk_w):
    """Gradient reaching the logits from an upstream gradient of the sigmoid router's top-k
    weights w_i = s_i / sum_chosen s: for a chosen expert e, dL/ds_e = (d_e - sum_i w_i d_i) /
    sum_chosen s, then dL/dz_e = s_e (1 - s_e) dL/ds_e; zero for the others."""
    s = _f64(s)
    idx = np.asarray(topk_idx, dtype=np.int64)
    d = _f64(d_topk_w)
    ss = np.take_along_axis(s, idx, axis=1)
    S = ss.sum(axis=1, keepdims=True)
    w = ss / S
    ds = (d - np.sum(w * d, axis=1, keepdims=True)) / S
    out = np.zeros_like(s)
    np.put_along_axis(out, idx, ss * (1.0 - ss) * ds, axis=1)
    return out


def bin_balance_grad_gate(g, topk_idx, expert_bin, n_bins, scale):
    """Gradient of scale * L_bal (eq. 16) with respect to the gate values g (f_e constant), the
    quantity bin_balance_grad_logits pushes through the softmax:
        dL/dg_je = N_B / |U_k| * (f_e - sum_{e' in B_k} f_e' h_je') / G_jk  (j in U_k, e in B_k)."""
    g = _f64(g)
    T, E = g.shape
    eb = np.asarray(expert_bin)
    N_B = E // n_bins
    _, parts = bin_balance_loss(g, topk_idx, expert_bin, n_bins)
    f = parts["f"]
    sel = np.zeros((T, E), dtype=bool)
    sel[np.arange(T)[:, None], np.asarray(topk_idx)] = True
    dg = np.zeros((T, E))
    for k in range(n_bins):
        if not parts["used"][k]:
            continue
        members = np.nonzero(eb == k)[0]
        U = sel[:, members].any(axis=1)
        gk = g[U][:, members]
        G = gk.sum(axis=1, keepdims=True)
        h = gk / G
        fk = f[members][None, :]
        dg[np.ix_(np.nonzero(U)[0], members)] = N_B / U.sum() * (fk - np.sum(fk * h, axis=1, keepdims=True)) / G
    return scale * dg


def bin_balance_grad_logits(z, topk_idx, expert_bin, n_bins, scale):
    """Gradient of scale * L_bal (eq. 16) at the gate logits z [T, E], with the routing
    fractions f_e held constant (they are counts; the gradient flows through P_e only, as for
    the standard load-balance loss). With h_je = g_je / G_jk, G_jk = sum_{e' in B_k} g_je' for a
    token j in U_k and e in B_k:
        dL/dg_je = N_B / |U_k| * (f_e - sum_{e' in B_k} f_e' h_je') / G_jk,
    then through the softmax: dz_je = g_je (dL/dg_je - sum_e' g_je' dL/dg_je')."""
    z = _f64(z)
    g = softmax_gate(z)
    T, E = g.shape
    eb = np.asarray(expert_bin)
    N_B = E // n_bins
    _, parts = bin_balance_loss(g, topk_idx, expert_bin, n_bins)
    f = parts["f"]
    sel = np.zeros((T, E), dtype=bool)
    sel[np.arange(T)[:, None], np.asarray(topk_idx)] = True
    dg = np.zeros((T, E))
    for k in range(n_bins):
        if not parts["used"][k]:
            continue
        members = np.nonzero(eb == k)[0]
        U = sel[:, members].any(axis=1)
        gk = g[U][:, members]
        G = gk.sum(axis=1, keepdims=True)
        h = gk / G
        fk = f[members][None, :]
        dg[np.ix_(np.nonzero(U)[0], members)] = N_B / U.sum() * (fk - np.sum(fk * h, axis=1, keepdims=True)) / G
    dg *= scale
    return g * (dg - np.sum(g * dg, axis=1, keepdims=True))
