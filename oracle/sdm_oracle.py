"""Float64 CPU oracle of the Sparse Delta Memory (SDM) hot path.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
module.  The CUDA library never calls it and shares no code with it.

What it computes, step by step, in the paper's order and notation
(arXiv 2607.07386):

1. Sparse key selection (Sec. 3.1 item 1; Sec. 2 "Product Key Memory"):
   pre-PKM scores s = P x in R^{2 sqrt(N)} (PROJECTED mode; DIRECT mode takes
   s = x), split into halves s1, s2 in R^{sqrt(N)}; the N slot scores are the
   outer sum s1 (+) s2 flattened row-major (slot = i*sqrt(N) + j); the top-k
   of the outer sum is taken as top_k(top_k(s1) (+) top_k(s2)) (Sec. 2).
   Selected scores are softmax-normalised (Sec. 4, "SDM Configuration") and the
   index list is sorted by slot (App. A.2, sort-by-index).
2. Learned initial state (Sec. 3.1, "Learned Initial State M0"): every
   sequence's memory starts as a copy of the per-head M0.
3. Gated delta write (Eqs. sdm-decay, sdm-write): for the write slots only,
   decay by alpha_t, then add beta_t * w_i * (v_t - v~_t) with the single
   prediction v~_t = sum_i w_i * M~_t[i]  (reading of Eq. sdm-write that makes
   the GDN reduction of Sec. 3.1 "Connection to GDN" exact; Fig. 1 draws the
   same data flow).  Unselected slots are unchanged (Sec. 3.1 item 2).
4. Sparse read (Eq. sdm-read) of the post-write memory M_t.

Precision: every input is the float64 value of its storage-dtype number.
Scores are accumulated in float64 in ascending d order (products of two bf16
or two fp32 numbers are exact in float64, so the only roundings are the
additions).  Rows written to memory and the output y are rounded to the
storage dtype (round-to-nearest-even, directly from float64); all other
intermediates stay in float64.

Tie-breaking (the paper is silent): per half by (score desc, index asc); over
the outer sum by (score desc, slot asc).

5. Lazy (copy-on-write) seeding of M0 (Sec. 3.1 "Learned Initial State"): the
   memory of a sequence is an overlay of the rows written so far over the
   read-only M0 of its head; a gather of a slot nobody has written returns the
   M0 row.  The results equal those of the copied memory of item 2.
6. Gate preparation and output epilogue around the path (Sec. 3.1, item 2 and
   "Norm, Gating, and Head Mixing"): alpha_t = exp(-A softplus(W_a x_t + b_dt)),
   beta_t = sigmoid(W_b x_t) per head; z = g (.) RMSNorm(y) per head, the heads
   concatenated per token and mixed by W_o.
7. The chunkwise (WY) form of the same recurrence (App. A.1-A.2): per chunk of C
   tokens, segmented cumulative log-decays, the gated sparse inner products A
   (write-write) and QK (read-write) by a two-pointer merge of sorted slot lists,
   a unit lower-triangular solve, then gather, correct, scatter and output against
   the chunk-initial memory.  Equal to item 3-4 up to rounding when the storage
   is exact; storage rounding is applied at chunk boundaries only.
8. The backward of the recurrence with in-place undo (App. A.3): the forward
   updates the memory in place and keeps, per token, the rows its write
   overwrote (O(T W d_v) beside the O(N d_v) memory); the backward walks the
   tokens in reverse, restores each token's pre-write rows from that log, and
   carries the adjoint of the memory for the touched rows only.  Gradients are
   those of the exact recurrence (storage rounding is not differentiated).
9. Access diagnostics (App. "Memory Utilization and Access"): the normalised
   effective number of keys exp(H(p)) / k, the cumulative mass curve C(m) of
   the descending-sorted weights, and the fraction of unique slots accessed.

Parity pins: see ``tests/test_oracle_pins.py`` (GDN reduction, dense masked
form, beta = 0 closed form, single-slot recall, brute-force top-k including
forced ties, invariants, the paper's state-size tables, lazy overlay against
the copied memory, diagnostics closed forms).
"""
from __future__ import annotations

import math

import numpy as np

__all__ = [
    "to_f64", "round_storage", "half_scores", "topk_half", "pkm_select", "address",
    "recur", "forward_slice", "state_elements_per_layer", "n_global_layers",
    "touched_mask", "recur_lazy", "materialize", "eff_keys_fraction", "cumulative_mass", "unique_fraction",
    "softplus", "gates", "norm_gate", "head_mix", "sparse_ip", "recur_chunkwise",
    "recur_forward_undo", "recur_backward", "round_e4m3", "quantize_undo", "undo_codes",
]


# --------------------------------------------------------------------------------------
# storage dtype helpers
# --------------------------------------------------------------------------------------

def to_f64(a: np.ndarray, dtype: str) -> np.ndarray:
    """Storage array -> float64 values.  "bf16" arrays hold the bfloat16 bit pattern
    as uint16; "f32" arrays are float32; "f64" arrays are returned as float64."""
    if dtype == "bf16":
        bits = np.asarray(a, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
        return bits.view(np.float32).astype(np.float64)
    return np.asarray(a, dtype=np.float64 if dtype == "f64" else np.float32).astype(np.float64)


def round_storage(x: np.ndarray, dtype: str) -> np.ndarray:
    """R(x): float64 -> nearest storage-dtype value (ties to even), returned as float64.

    bf16 has 8 significant bits: the value is snapped to the multiple of
    2^(e-8) nearest to x, where 2^(e-1) <= |x| < 2^e (quantum clamped at the
    subnormal step 2^-133).  "f64" is the identity (exact storage, used by pins).
    """
    x = np.asarray(x, dtype=np.float64)
    if dtype == "f64":
        return x.copy()
    if dtype == "f32":
        return x.astype(np.float32).astype(np.float64)
    if dtype != "bf16":
        raise ValueError(dtype)
    _, e = np.frexp(x)
    step = np.ldexp(1.0, np.maximum(e - 8, -133))
    return np.rint(x / step) * step


def to_bf16_bits(x64: np.ndarray) -> np.ndarray:
    """Bit pattern of the bf16 numbers R(x) (x already representable)."""
    return (np.asarray(x64, np.float64).astype(np.float32).view(np.uint32) >> np.uint32(16)).astype(np.uint16)


# --------------------------------------------------------------------------------------
# addressing (Sec. 2 Product Key Memory; Sec. 3.1 item 1)
# --------------------------------------------------------------------------------------

def half_scores(P: np.ndarray | None, X: np.ndarray) -> np.ndarray:
    """Pre-PKM scores s = P x for every token.

    P: [2S, d_k] float64 (None for DIRECT mode, where s = x), X: [T, d_k] float64.
    Returns [T, 2S] float64, each entry summed over d = 0, 1, ..., d_k-1 in that order.
    """
    if P is None:
        return np.array(X, dtype=np.float64, copy=True)
    s = np.zeros((X.shape[0], P.shape[0]), dtype=np.float64)
    for d in range(P.shape[1]):
        s += X[:, d:d + 1] * P[None, :, d]
    return s


def topk_half(s: np.ndarray, k: int) -> np.ndarray:
    """Indices of the top-k of each row of s under (value desc, index asc), best first."""
    order = np.argsort(-s, axis=-1, kind="stable")
    return order[..., :k]


def pkm_select(s1: np.ndarray, s2: np.ndarray, k: int):
    """top_k(top_k(s1) (+) top_k(s2)) for every token (Sec. 2, PKM identity).

    s1, s2: [T, S].  Returns (idx [T, k] int64 sorted ascending by slot,
    score [T, k] float64 combined scores in the same order, w [T, k] softmax weights).
    Candidate order: (score desc, slot asc); slot = i * S + j (row-major outer sum).
    """
    T, S = s1.shape
    i1 = topk_half(s1, k)                                   # [T, k]
    i2 = topk_half(s2, k)
    v1 = np.take_along_axis(s1, i1, axis=1)
    v2 = np.take_along_axis(s2, i2, axis=1)
    cand = (v1[:, :, None] + v2[:, None, :]).reshape(T, k * k)
    slot = (i1[:, :, None] * S + i2[:, None, :]).reshape(T, k * k)
    pick = np.lexsort((slot, -cand), axis=-1)[:, :k]        # primary: score desc; then slot asc
    sel_slot = np.take_along_axis(slot, pick, axis=1)
    sel_score = np.take_along_axis(cand, pick, axis=1)
    by_slot = np.argsort(sel_slot, axis=1, kind="stable")
    idx = np.take_along_axis(sel_slot, by_slot, axis=1)
    score = np.take_along_axis(sel_score, by_slot, axis=1)
    z = np.exp(score - score.max(axis=1, keepdims=True))
    w = z / z.sum(axis=1, keepdims=True)
    return idx, score, w


def address(P: np.ndarray | None, X: np.ndarray, N: int, k: int, block: int = 2048):
    """Sparse key selection for every token of one head: (idx, score, w), each [T, k].
    Tokens are independent; they are processed in blocks only to bound memory."""
    S = math.isqrt(N)
    assert S * S == N
    parts = []
    for t0 in range(0, X.shape[0], block):
        s = half_scores(P, X[t0:t0 + block])
        assert s.shape[1] == 2 * S, "scores must have 2 sqrt(N) entries"
        parts.append(pkm_select(s[:, :S], s[:, S:], k))
    if not parts:
        z = np.zeros((0, k))
        return z.astype(np.int64), z, z
    return tuple(np.concatenate([p[i] for p in parts]) for i in range(3))


# --------------------------------------------------------------------------------------
# recurrence (Eqs. sdm-decay, sdm-write, sdm-read)
# --------------------------------------------------------------------------------------

def recur(M: np.ndarray, idx_w, w_w, idx_r, w_r, v, alpha, beta, store: str):
    """Run the sparse gated delta recurrence over T tokens of one (b, h) slice.

    M: [N, d_v] float64 memory, updated in place (values stay representable in
    the storage dtype).  idx_*: [T, k_*] int, w_*: [T, k_*] float64,
    v: [T, d_v], alpha, beta: [T] (float64).  Within a token the write slots
    must be distinct.  Returns (y [T, d_v] float64 before rounding, R(y)).
    """
    T = v.shape[0]
    y = np.empty((T, M.shape[1]), dtype=np.float64)
    for t in range(T):
        iw = idx_w[t]
        decayed = alpha[t] * M[iw]                  # M~_t[i] = alpha_t M_{t-1}[i], i in I^w_t   (Eq. sdm-decay)
        pred = w_w[t] @ decayed                     # v~_t = sum_i k_t^(i) M~_t[i]
        delta = v[t] - pred                         # v_t - v~_t
        M[iw] = round_storage(decayed + beta[t] * w_w[t][:, None] * delta[None, :], store)  # Eq. sdm-write
        y[t] = w_r[t] @ M[idx_r[t]]                 # y_t = sum_i q_t^(i) M_t[i]   (Eq. sdm-read, post-write)
    return y, round_storage(y, store)


def forward_slice(M0_h: np.ndarray, P_q, P_k, q, k, v, alpha, beta, N: int, k_write: int, k_read: int,
                  store: str, M: np.ndarray | None = None):
    """Whole hot path for one (b, h) slice, all inputs already float64.

    M0_h: [N, d_v] initial memory of head h (copied: Sec. 3.1 "Learned Initial
    State"), unless a running memory M is given (continuing a sequence).
    Returns dict with y (rounded), y64, M (final memory), idx_w, w_w, idx_r, w_r.
    """
    idx_w, _, w_w = address(P_k, k, N, k_write)
    idx_r, _, w_r = address(P_q, q, N, k_read)
    if M is None:
        M = np.array(M0_h, dtype=np.float64, copy=True)
    y64, y = recur(M, idx_w, w_w, idx_r, w_r, v, alpha, beta, store)
    return {"y": y, "y64": y64, "M": M, "idx_w": idx_w, "w_w": w_w, "idx_r": idx_r, "w_r": w_r}


# --------------------------------------------------------------------------------------
# chunkwise (WY) form (App. A.1 "Intra-Chunk Parallel vs. Chunkwise Recurrent", A.2)
# --------------------------------------------------------------------------------------

def sparse_ip(idx_a, val_a, lam_a, idx_b, val_b, lam_b) -> float:
    """Gated sparse inner product of two tokens (App. A.2, Eq. sparse-ip):
    sum over matching slots idx_a[n] == idx_b[m] of val_a[n] val_b[m] exp(lam_a[n] - lam_b[m]).
    Both index lists must be strictly ascending; they are walked together (two pointers)."""
    total = 0.0
    a = b = 0
    while a < len(idx_a) and b < len(idx_b):
        ia, ib = idx_a[a], idx_b[b]
        if ia == ib:
            total += val_a[a] * val_b[b] * math.exp(lam_a[a] - lam_b[b])
            a += 1
            b += 1
        elif ia < ib:
            a += 1
        else:
            b += 1
    return total


def recur_chunkwise(M: np.ndarray, idx_w, w_w, idx_r, w_r, v, alpha, beta, C: int, store: str):
    """The recurrence of ``recur`` in chunkwise form (App. A.1-A.2), chunks of C tokens.

    Phase 1 (per chunk, independent of the memory): lam_w[t, n], the cumulative log-decay of
    slot idx_w[t, n] over the chunk's writers of that slot up to and including t; lam_r[t, n]
    the same for read slot idx_r[t, n] after token t's own write; the lower-triangular
    A[t, s] = sparse_ip(write t, write s) for s < t and QK[t, s] = sparse_ip(read t, write s)
    for s <= t; M_sys = I + diag(beta) A; dV_const = M_sys^-1 diag(beta) V and
    B = M_sys^-1 diag(-beta).
    Phase 2 (sequential over chunks): retrieved[t] = sum_n w e^lam_w M[idx_w[t, n]] and
    inter[t] = sum_n rho e^lam_r M[idx_r[t, n]] from the chunk-initial memory; the written
    deltas u = dV_const + B retrieved (u_t = beta_t (v_t - v~_t)); y = inter + QK u; then
    every written slot i becomes e^(lam_i) M[i] + sum_t e^(lam_i - lam_(t,i)) w_(t,i) u_t with
    lam_i its decay over the whole chunk, rounded to the storage dtype.

    M: [N, d_v] float64, updated in place.  Returns (y [T, d_v] float64, R(y)).
    """
    from scipy.linalg import solve_triangular
    T = v.shape[0]
    y = np.empty((T, M.shape[1]), dtype=np.float64)
    for c0 in range(0, T, C):
        c1 = min(T, c0 + C)
        n = c1 - c0
        # ---- phase 1: segmented cumulative log-decay, interaction matrices, triangular solve
        acc = {}
        lam_w = np.zeros(idx_w[c0:c1].shape)
        lam_r = np.zeros(idx_r[c0:c1].shape)
        for t in range(n):
            la = math.log(alpha[c0 + t])
            for m, i in enumerate(idx_w[c0 + t]):
                acc[int(i)] = acc.get(int(i), 0.0) + la
                lam_w[t, m] = acc[int(i)]
            for m, j in enumerate(idx_r[c0 + t]):
                lam_r[t, m] = acc.get(int(j), 0.0)
        A = np.zeros((n, n))
        QK = np.zeros((n, n))
        for t in range(n):
            for s_ in range(n):
                if s_ < t:
                    A[t, s_] = sparse_ip(idx_w[c0 + t], w_w[c0 + t], lam_w[t], idx_w[c0 + s_], w_w[c0 + s_], lam_w[s_])
                if s_ <= t:
                    QK[t, s_] = sparse_ip(idx_r[c0 + t], w_r[c0 + t], lam_r[t], idx_w[c0 + s_], w_w[c0 + s_], lam_w[s_])
        bet = np.asarray(beta[c0:c1], dtype=np.float64)
        M_sys = np.eye(n) + bet[:, None] * A
        dV_const = solve_triangular(M_sys, bet[:, None] * v[c0:c1], lower=True, unit_diagonal=True)
        Bm = solve_triangular(M_sys, np.diag(-bet), lower=True, unit_diagonal=True)
        # ---- phase 2: gather, correct, output, scatter
        retrieved = np.stack([(w_w[c0 + t] * np.exp(lam_w[t])) @ M[idx_w[c0 + t]] for t in range(n)])
        inter = np.stack([(w_r[c0 + t] * np.exp(lam_r[t])) @ M[idx_r[c0 + t]] for t in range(n)])
        u = dV_const + Bm @ retrieved
        y[c0:c1] = inter + QK @ u
        touched = sorted(acc)
        new = {i: math.exp(acc[i]) * M[i] for i in touched}
        for t in range(n):
            for m, i in enumerate(idx_w[c0 + t]):
                i = int(i)
                new[i] = new[i] + math.exp(acc[i] - lam_w[t, m]) * w_w[c0 + t][m] * u[t]
        for i in touched:
            M[i] = round_storage(new[i], store)
    return y, round_storage(y, store)


# --------------------------------------------------------------------------------------
# backward with in-place undo (App. A.3 "Memory-Efficient Backward")
# --------------------------------------------------------------------------------------

def recur_forward_undo(M: np.ndarray, idx_w, w_w, idx_r, w_r, v, alpha, beta, store: str = "f64"):
    """``recur`` that also returns the undo log: for every token, the rows M_{t-1}[I^w_t] its
    write overwrote (stored values).  M is updated in place to M_T; written rows are rounded to
    ``store``.  Returns (y [T, d_v] float64 from the stored rows, undo [T, k_w, d_v])."""
    T = v.shape[0]
    y = np.empty((T, M.shape[1]))
    undo = np.empty((T, idx_w.shape[1], M.shape[1]))
    for t in range(T):
        iw = idx_w[t]
        undo[t] = M[iw]
        decayed = alpha[t] * M[iw]
        delta = v[t] - w_w[t] @ decayed
        M[iw] = round_storage(decayed + beta[t] * w_w[t][:, None] * delta[None, :], store)
        y[t] = w_r[t] @ M[idx_r[t]]
    return y, undo


def recur_backward(M: np.ndarray, undo, idx_w, w_w, idx_r, w_r, v, alpha, beta, dy):
    """Reverse-mode gradients of sum_t <dy_t, y_t> through the recurrence, from the final memory
    M (= M_T, restored in place to M_0 on return) and the undo log of ``recur_forward_undo``.

    Token t, in reverse: the read y_t = sum_n rho_n M_t[r_n] gives d rho_n = <dy_t, M_t[r_n]> and
    adds rho_n dy_t to the memory adjoint G at r_n.  The write M_t[i] = r_i + beta w_i delta with
    r_i = alpha M_{t-1}[i] and delta = v_t - sum_m w_m r_m gives, with G_i the adjoint of M_t[i]:
    d delta = beta sum_i w_i G_i, d beta = sum_i w_i <G_i, delta>, d w_i = beta <G_i, delta> -
    <r_i, d delta>, d v_t = d delta, d r_i = G_i - w_i d delta, d alpha = sum_i <d r_i, M_{t-1}[i]>,
    and the adjoint of M_{t-1}[i] becomes alpha d r_i.  M_{t-1}[I^w_t] comes back from the log.

    Returns dict: dv [T, d_v], dalpha [T], dbeta [T], dw_w [T, k_w], dw_r [T, k_r], dM0 [N, d_v].
    """
    T, dvdim = v.shape
    G = {}
    out = {"dv": np.zeros_like(v), "dalpha": np.zeros(T), "dbeta": np.zeros(T),
           "dw_w": np.zeros(w_w.shape), "dw_r": np.zeros(w_r.shape)}
    zero = np.zeros(dvdim)
    for t in range(T - 1, -1, -1):
        # read of the post-write memory M_t
        for n, j in enumerate(idx_r[t]):
            j = int(j)
            out["dw_r"][t, n] = dy[t] @ M[j]
            G[j] = G.get(j, zero) + w_r[t][n] * dy[t]
        # write: recover M_{t-1} on the written rows, then the chain rule through the update
        iw = [int(i) for i in idx_w[t]]
        prev = undo[t]
        r = alpha[t] * prev
        delta = v[t] - w_w[t] @ r
        Gi = np.stack([G.get(i, zero) for i in iw])
        d_delta = beta[t] * (w_w[t] @ Gi)
        out["dbeta"][t] = np.sum(w_w[t] * (Gi @ delta))
        out["dw_w"][t] = beta[t] * (Gi @ delta) - r @ d_delta
        out["dv"][t] = d_delta
        d_r = Gi - w_w[t][:, None] * d_delta[None, :]
        out["dalpha"][t] = np.sum(d_r * prev)
        for m, i in enumerate(iw):
            G[i] = alpha[t] * d_r[m]
            M[i] = prev[m]                           # undo: M_t[i] -> M_{t-1}[i]
    dM0 = np.zeros_like(M)
    for i, g in G.items():
        dM0[i] = g
    out["dM0"] = dM0
    return out


def round_e4m3(x: np.ndarray) -> np.ndarray:
    """Nearest fp8 e4m3 value (ties to even) of x, |x| <= 448: 4 significant bits for
    |x| >= 2^-6, a fixed step of 2^-9 below (subnormals)."""
    x = np.asarray(x, dtype=np.float64)
    _, e = np.frexp(x)
    q = np.ldexp(1.0, np.maximum(e - 4, -9))
    return np.rint(x / q) * q


def quantize_undo(undo: np.ndarray, kind: str, arith: str = "f64") -> np.ndarray:
    """The undo log as a quantised snapshot would give it back (App. A.3: fp8 or int4 snapshots
    for long sequences), one scale per logged row: "fp8" rounds row / s to e4m3 with
    s = max|row| / 448; "int4" rounds row / s to the integers -7..7 with s = max|row| / 7;
    "exact" returns the log unchanged.

    arith="f64" does the arithmetic in float64.  arith="f32" takes every step in float32 with
    correctly rounded operations (the scale, the division by it and the dequantising product
    q * s), so that the codes are decided in the precision a float32 implementation uses:
    the values equal ``undo_codes``' codes times their scales, rounded to float32."""
    u = np.asarray(undo, dtype=np.float64)
    if kind == "exact":
        return u.copy()
    if arith == "f32":
        codes, scale = undo_codes(u, kind)
        return (codes.astype(np.float32) * scale[..., None]).astype(np.float64)
    top = {"fp8": 448.0, "int4": 7.0}[kind]
    amax = np.max(np.abs(u), axis=-1, keepdims=True)
    scale = np.where(amax > 0, amax / top, 1.0)
    y = u / scale
    q = round_e4m3(y) if kind == "fp8" else np.clip(np.rint(y), -7, 7)
    return q * scale


def undo_codes(undo: np.ndarray, kind: str):
    """The quantised snapshot itself, in float32 arithmetic: per logged row the scale
    s = fl32(max|row| / top) (1 for an all-zero row) and the codes q = round(fl32(row / s)),
    e4m3 values for "fp8" (top 448, ties to even) and integers -7..7 for "int4" (top 7, ties
    to even).  The rows must be float32-representable (stored values).  Returns (codes as
    float64 [..., d_v], scales as float32 [...])."""
    u = np.asarray(undo, dtype=np.float64)
    u32 = u.astype(np.float32)
    if not np.array_equal(u32.astype(np.float64), u):
        raise ValueError("undo_codes: the logged rows must be float32 values")
    top = np.float32({"fp8": 448.0, "int4": 7.0}[kind])
    amax = np.max(np.abs(u32), axis=-1)
    scale = np.where(amax > 0, amax / top, np.float32(1.0)).astype(np.float32)
    y = (u32 / scale[..., None]).astype(np.float32).astype(np.float64)
    q = round_e4m3(np.clip(y, -448.0, 448.0)) if kind == "fp8" else np.clip(np.rint(y), -7, 7)
    return q, scale


# --------------------------------------------------------------------------------------
# lazy (copy-on-write) initial state (Sec. 3.1 "Learned Initial State M0")
# --------------------------------------------------------------------------------------

def touched_mask(idx_w: np.ndarray, N: int, prior: np.ndarray | None = None) -> np.ndarray:
    """Boolean [N]: slots written by any token of idx_w ([T, k_write]), or already marked in prior."""
    m = np.zeros(N, dtype=bool) if prior is None else np.array(prior, dtype=bool, copy=True)
    m[np.asarray(idx_w, dtype=np.int64).ravel()] = True
    return m


def recur_lazy(M0_h: np.ndarray, overlay: dict, idx_w, w_w, idx_r, w_r, v, alpha, beta, store: str):
    """The recurrence of ``recur`` on a copy-on-write memory: ``overlay`` maps slot -> row
    (float64) for the slots written so far and is updated in place; every other slot reads
    M0_h (never modified).  Returns (y64, R(y)) like ``recur``."""
    def row(s):
        return overlay[s] if s in overlay else M0_h[s]
    T = v.shape[0]
    y = np.empty((T, M0_h.shape[1]), dtype=np.float64)
    for t in range(T):
        iw = [int(s) for s in idx_w[t]]
        decayed = [alpha[t] * row(s) for s in iw]                       # Eq. sdm-decay
        pred = sum(w_w[t][n] * decayed[n] for n in range(len(iw)))      # v~_t
        delta = v[t] - pred
        for n, s in enumerate(iw):                                      # Eq. sdm-write
            overlay[s] = round_storage(decayed[n] + beta[t] * w_w[t][n] * delta, store)
        y[t] = sum(w_r[t][n] * row(int(s)) for n, s in enumerate(idx_r[t]))   # Eq. sdm-read
    return y, round_storage(y, store)


def materialize(M0_h: np.ndarray, overlay: dict) -> np.ndarray:
    """Dense memory of a copy-on-write state: M0_h with the overlay's rows in place."""
    M = np.array(M0_h, dtype=np.float64, copy=True)
    for s, r in overlay.items():
        M[s] = r
    return M


# --------------------------------------------------------------------------------------
# access diagnostics (App. "Memory Utilization and Access")
# --------------------------------------------------------------------------------------

def eff_keys_fraction(p: np.ndarray) -> np.ndarray:
    """u(p) = exp(H(p)) / k per token, H(p) = -sum_i p_i log p_i (0 log 0 = 0); p: [..., k]."""
    p = np.asarray(p, dtype=np.float64)
    plogp = np.where(p > 0, p * np.log(np.where(p > 0, p, 1.0)), 0.0)
    return np.exp(-plogp.sum(axis=-1)) / p.shape[-1]


def cumulative_mass(p: np.ndarray) -> np.ndarray:
    """C(m) = sum of the m largest weights, m = 1..k, per token; p: [..., k] -> [..., k]."""
    p = np.asarray(p, dtype=np.float64)
    return np.cumsum(-np.sort(-p, axis=-1), axis=-1)


def unique_fraction(idx: np.ndarray, N: int) -> float:
    """Fraction of the N slots that appear in idx (any shape)."""
    return np.unique(np.asarray(idx, dtype=np.int64)).size / N


# --------------------------------------------------------------------------------------
# gate preparation and output epilogue (Sec. 3.1)
# --------------------------------------------------------------------------------------

def softplus(z: np.ndarray) -> np.ndarray:
    """softplus(z) = log(1 + e^z), evaluated as logaddexp(0, z) (no overflow)."""
    return np.logaddexp(0.0, np.asarray(z, dtype=np.float64))


def gates(x: np.ndarray, W_a: np.ndarray, b_dt: np.ndarray, A: np.ndarray, W_b: np.ndarray):
    """Per-head forget and input gates of every token (Sec. 3.1, after Eq. sdm-write):
    alpha_t = exp(-A softplus(W_a x_t + b_dt)), beta_t = sigmoid(W_b x_t).

    x: [T, d]; W_a, W_b: [H, d]; b_dt, A: [H].  Returns (alpha, beta), each [H, T] float64.
    """
    x = np.asarray(x, dtype=np.float64)
    za = x @ np.asarray(W_a, dtype=np.float64).T + np.asarray(b_dt, dtype=np.float64)[None, :]
    zb = x @ np.asarray(W_b, dtype=np.float64).T
    alpha = np.exp(-np.asarray(A, dtype=np.float64)[None, :] * softplus(za))
    beta = 1.0 / (1.0 + np.exp(-zb))
    return alpha.T, beta.T


def norm_gate(y: np.ndarray, g: np.ndarray, gamma: np.ndarray, eps: float) -> np.ndarray:
    """g (.) RMSNorm(y) for one head (Sec. 3.1 "Norm, Gating, and Head Mixing"):
    y, g: [T, d_v]; gamma: [d_v] RMSNorm scale; returns g * gamma * y / sqrt(mean(y^2) + eps)."""
    y = np.asarray(y, dtype=np.float64)
    rms = np.sqrt(np.mean(y * y, axis=-1, keepdims=True) + eps)
    return np.asarray(g, dtype=np.float64) * np.asarray(gamma, dtype=np.float64)[None, :] * y / rms


def head_mix(z: np.ndarray, W_o: np.ndarray) -> np.ndarray:
    """Output projection mixing the heads: z [H, T, d_v] -> o [T, d] = concat_h(z_h) W_o^T,
    W_o: [d, H * d_v] (head h owns columns h*d_v .. (h+1)*d_v - 1)."""
    H, T, dv = z.shape
    zt = np.transpose(np.asarray(z, dtype=np.float64), (1, 0, 2)).reshape(T, H * dv)
    return zt @ np.asarray(W_o, dtype=np.float64).T


# --------------------------------------------------------------------------------------
# geometry (Sec. 3.2 / 3.3, Sec. 4 "SDM Configuration")
# --------------------------------------------------------------------------------------

def n_global_layers(layers: int) -> int:
    """Global (long-range) layers in the 3:1 local:global hybrid (Sec. 4, Architecture)."""
    return layers // 4


def state_elements_per_layer(d: int, H: int) -> int:
    """SDM state of one layer: H heads x N slots x d_v, with N = (d / 4H)^2 and d_v = d / H
    (Sec. 4 "SDM Configuration"; d_qk^total = d/2 and d_v^total = d from Sec. 3.2, Eq. of Sec. 3.3)."""
    assert d % (4 * H) == 0
    n = (d // (4 * H)) ** 2
    return H * n * (d // H)
