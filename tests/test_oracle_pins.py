"""Pins of the float64 oracle against facts fixed by the paper and by mathematics.

Each test checks the oracle against something other than itself: a textbook
formula (Gated DeltaNet, Eq. gdn-update), an independent dense formulation of
the sparse update, a closed form, brute force over all N slots, a library
routine (bf16 rounding in torch, a BLAS matmul), or numbers printed in the
paper (Table 1, Table 3, App. A.3).  The last tests plant plausible mistakes
in copies of the oracle and check that a pin rejects each.
"""
import math
import os

import numpy as np
import pytest

from oracle import sdm_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden_rows(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                rows.append(line.split())
    return rows


# ------------------------------------------------------------------ storage rounding

def test_bf16_rounding_matches_torch_on_fp32_values():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(7)
    x32 = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-6, 6, 20000),
                          np.float32(1.0) + np.arange(-64, 64) * np.float32(2.0 ** -9)]).astype(np.float32)
    ref = torch.from_numpy(x32).to(torch.bfloat16).to(torch.float64).numpy()
    got = O.round_storage(x32.astype(np.float64), "bf16")
    assert np.array_equal(got, ref)


def test_bf16_rounding_is_direct_from_float64():
    # Just above the midpoint between 1 and 1+2^-7: nearest bf16 is 1+2^-7.
    # Rounding through fp32 first would land exactly on the midpoint and then tie to 1.0.
    x = 1.0 + 2.0 ** -8 + 2.0 ** -30
    assert O.round_storage(np.array([x]), "bf16")[0] == 1.0 + 2.0 ** -7
    assert O.round_storage(np.array([1.0 + 2.0 ** -8]), "bf16")[0] == 1.0          # tie -> even
    assert O.round_storage(np.array([1.0 + 3 * 2.0 ** -8]), "bf16")[0] == 1.0 + 2.0 ** -6
    bits = O.to_bf16_bits(O.round_storage(np.array([-2.5, 1.0, 0.0]), "bf16"))
    assert list(bits) == [0xC020, 0x3F80, 0x0000]


# ------------------------------------------------------------------ addressing

def test_half_scores_against_matmul_and_exact_integers():
    rng = np.random.default_rng(1)
    P = rng.standard_normal((32, 24))
    X = rng.standard_normal((5, 24))
    np.testing.assert_allclose(O.half_scores(P, X), X @ P.T, rtol=1e-13, atol=1e-13)
    Pi = rng.integers(-9, 10, (32, 24)).astype(np.float64)
    Xi = rng.integers(-9, 10, (5, 24)).astype(np.float64)
    assert np.array_equal(O.half_scores(Pi, Xi), (Xi.astype(np.int64) @ Pi.astype(np.int64).T).astype(np.float64))
    assert np.array_equal(O.half_scores(None, Xi), Xi)


def _brute_topk(s1, s2, k):
    """Exact top-k over all N = S*S flattened outer-sum scores, (score desc, slot asc)."""
    S = s1.shape[0]
    full = (s1[:, None] + s2[None, :]).reshape(-1)
    slot = np.arange(S * S)
    pick = np.lexsort((slot, -full))[:k]
    return np.sort(slot[pick])


@pytest.mark.parametrize("S,k,integer", [(8, 3, False), (16, 8, False), (16, 8, True), (32, 16, True),
                                         (8, 8, True), (64, 8, False), (5, 5, True), (1, 1, False),
                                         (2, 2, True), (3, 1, True)])
def test_pkm_two_stage_equals_brute_force(S, k, integer):
    rng = np.random.default_rng(S * 100 + k)
    T = 200
    if integer:   # few distinct values: many exact ties in both halves and in the outer sum
        s1 = rng.integers(-3, 4, (T, S)).astype(np.float64)
        s2 = rng.integers(-3, 4, (T, S)).astype(np.float64)
    else:
        s1 = rng.standard_normal((T, S))
        s2 = rng.standard_normal((T, S))
    idx, score, w = O.pkm_select(s1, s2, k)
    for t in range(T):
        assert np.array_equal(idx[t], _brute_topk(s1[t], s2[t], k)), t
        assert np.all(np.diff(idx[t]) > 0)
        np.testing.assert_array_equal(score[t], s1[t][idx[t] // S] + s2[t][idx[t] % S])
    np.testing.assert_allclose(w.sum(axis=1), 1.0, rtol=0, atol=1e-14)
    ref_w = np.exp(score) / np.exp(score).sum(axis=1, keepdims=True)
    np.testing.assert_allclose(w, ref_w, rtol=1e-12)


def test_address_projected_end_to_end_brute_force():
    rng = np.random.default_rng(3)
    S, dk, k, T = 16, 12, 6, 50
    P = rng.standard_normal((2 * S, dk))
    X = rng.standard_normal((T, dk))
    idx, _, _ = O.address(P, X, S * S, k)
    s = X @ P.T
    for t in range(T):
        assert np.array_equal(idx[t], _brute_topk(s[t, :S], s[t, S:], k))


def test_address_of_no_tokens_is_empty():
    P = np.ones((8, 3))
    idx, score, w = O.address(P, np.zeros((0, 3)), 16, 2)
    assert idx.shape == (0, 2) and score.shape == (0, 2) and w.shape == (0, 2)


def test_address_direct_mode_uses_x_halves():
    rng = np.random.default_rng(4)
    S, k = 8, 4
    X = rng.standard_normal((10, 2 * S))
    idx, _, _ = O.address(None, X, S * S, k)
    for t in range(10):
        assert np.array_equal(idx[t], _brute_topk(X[t, :S], X[t, S:], k))


# ------------------------------------------------------------------ recurrence

def _gdn_textbook(M, K, V, Q, alpha, beta):
    """Gated DeltaNet (Eq. gdn-update): M_t = a M + b k (v - a M^T k)^T, read y = M_t^T q."""
    M = M.copy()
    ys = []
    for t in range(K.shape[0]):
        k, v, q = K[t], V[t], Q[t]
        M = alpha[t] * M + beta[t] * np.outer(k, v - alpha[t] * (M.T @ k))
        ys.append(M.T @ q)
    return M, np.array(ys)


def test_gdn_reduction_all_slots_dense_keys():
    """Sec. 3.1 "Connection to GDN": N = d_qk, W = R = N, dense key values -> GDN exactly."""
    rng = np.random.default_rng(11)
    dqk, dv, T = 6, 5, 40
    M0 = rng.standard_normal((dqk, dv))
    K = rng.standard_normal((T, dqk)) / np.sqrt(dqk)
    Q = rng.standard_normal((T, dqk))
    V = rng.standard_normal((T, dv))
    alpha = 1 / (1 + np.exp(-rng.standard_normal(T) - 2))
    beta = 1 / (1 + np.exp(-rng.standard_normal(T)))
    allslots = np.tile(np.arange(dqk), (T, 1))
    M = M0.copy()
    y64, _ = O.recur(M, allslots, K, allslots, Q, V, alpha, beta, "f64")
    M_ref, y_ref = _gdn_textbook(M0, K, V, Q, alpha, beta)
    np.testing.assert_allclose(M, M_ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(y64, y_ref, rtol=1e-12, atol=1e-12)


def _dense_masked_sdm(M0, idx_w, w_w, idx_r, w_r, V, alpha, beta):
    """The same update written densely over all N slots: decay mask D_t = I + (a-1) diag(1[i in I^w]),
    dense write vector kappa (zero off I^w), dense read vector rho (zero off I^r)."""
    N = M0.shape[0]
    M = M0.copy()
    ys = []
    for t in range(V.shape[0]):
        mask = np.zeros(N)
        mask[idx_w[t]] = 1.0
        kappa = np.zeros(N)
        kappa[idx_w[t]] = w_w[t]
        rho = np.zeros(N)
        rho[idx_r[t]] = w_r[t]
        Mt = (1.0 + (alpha[t] - 1.0) * mask)[:, None] * M
        Mt = Mt + beta[t] * np.outer(kappa, V[t] - Mt.T @ kappa)
        M = Mt
        ys.append(M.T @ rho)
    return M, np.array(ys)


def _random_sparse_case(rng, N=40, dv=4, T=60, kw=5, kr=4):
    idx_w = np.array([np.sort(rng.choice(N, kw, replace=False)) for _ in range(T)])
    idx_r = np.array([np.sort(rng.choice(N, kr, replace=False)) for _ in range(T)])
    w_w = rng.dirichlet(np.ones(kw), T)
    w_r = rng.dirichlet(np.ones(kr), T)
    V = rng.standard_normal((T, dv))
    alpha = 1 / (1 + np.exp(-rng.standard_normal(T) - 1))
    beta = 1 / (1 + np.exp(-rng.standard_normal(T)))
    M0 = rng.standard_normal((N, dv))
    return M0, idx_w, w_w, idx_r, w_r, V, alpha, beta


def test_sparse_recurrence_equals_dense_masked_form():
    rng = np.random.default_rng(12)
    M0, idx_w, w_w, idx_r, w_r, V, alpha, beta = _random_sparse_case(rng)
    M = M0.copy()
    y64, _ = O.recur(M, idx_w, w_w, idx_r, w_r, V, alpha, beta, "f64")
    M_ref, y_ref = _dense_masked_sdm(M0, idx_w, w_w, idx_r, w_r, V, alpha, beta)
    np.testing.assert_allclose(M, M_ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(y64, y_ref, rtol=1e-12, atol=1e-12)


def test_beta_zero_closed_form():
    """beta = 0: a slot only decays, by the product of alpha over the tokens that write it."""
    rng = np.random.default_rng(13)
    M0, idx_w, w_w, idx_r, w_r, V, alpha, _ = _random_sparse_case(rng)
    T, N = V.shape[0], M0.shape[0]
    M = M0.copy()
    y64, _ = O.recur(M, idx_w, w_w, idx_r, w_r, V, alpha, np.zeros(T), "f64")
    decay = np.ones(N)
    for t in range(T):
        decay[idx_w[t]] *= alpha[t]
        np.testing.assert_allclose(y64[t], w_r[t] @ (decay[idx_r[t], None] * M0[idx_r[t]]), rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(M, decay[:, None] * M0, rtol=1e-13, atol=1e-15)


@pytest.mark.parametrize("store", ["bf16", "f32", "f64"])
def test_single_slot_recall_exact(store):
    """alpha = beta = 1, one slot per token (softmax weight exactly 1): the slot becomes v_t and
    reading it returns v_t, bit for bit in the storage dtype."""
    rng = np.random.default_rng(14)
    N, dv, T = 64, 16, 30
    M0 = O.round_storage(rng.standard_normal((N, dv)), store)
    V = O.round_storage(rng.standard_normal((T, dv)), store)
    slots = rng.choice(N, T, replace=False)[:, None]
    M = M0.copy()
    _, y = O.recur(M, slots, np.ones((T, 1)), slots, np.ones((T, 1)), V, np.ones(T), np.ones(T), store)
    if store == "f64":   # r + (v - r) is only exact when v and r carry few significant bits
        np.testing.assert_allclose(y, V, rtol=1e-15, atol=1e-15)
        np.testing.assert_allclose(M[slots[:, 0]], V, rtol=1e-15, atol=1e-15)
    else:
        assert np.array_equal(y, V)
        assert np.array_equal(M[slots[:, 0]], V)
    untouched = np.setdiff1d(np.arange(N), slots[:, 0])
    assert np.array_equal(M[untouched], M0[untouched])


def test_untouched_rows_bit_identical_and_split_invariance():
    rng = np.random.default_rng(15)
    M0, idx_w, w_w, idx_r, w_r, V, alpha, beta = _random_sparse_case(rng, N=500, T=80)
    M0 = O.round_storage(M0 * 0.02, "bf16")
    V = O.round_storage(V, "bf16")
    Ma = M0.copy()
    _, ya = O.recur(Ma, idx_w, w_w, idx_r, w_r, V, alpha, beta, "bf16")
    Mb = M0.copy()
    _, yb1 = O.recur(Mb, idx_w[:33], w_w[:33], idx_r[:33], w_r[:33], V[:33], alpha[:33], beta[:33], "bf16")
    _, yb2 = O.recur(Mb, idx_w[33:], w_w[33:], idx_r[33:], w_r[33:], V[33:], alpha[33:], beta[33:], "bf16")
    assert np.array_equal(Ma, Mb) and np.array_equal(ya, np.concatenate([yb1, yb2]))
    untouched = np.setdiff1d(np.arange(500), idx_w.ravel())
    assert untouched.size > 0 and np.array_equal(Ma[untouched], M0[untouched])
    assert np.array_equal(O.round_storage(Ma, "bf16"), Ma)


def test_forward_slice_is_address_then_recur():
    rng = np.random.default_rng(16)
    S, dk, dv, T, k = 8, 10, 6, 40, 4
    N = S * S
    Pq, Pk = rng.standard_normal((2 * S, dk)), rng.standard_normal((2 * S, dk))
    q, kk, v = rng.standard_normal((T, dk)), rng.standard_normal((T, dk)), rng.standard_normal((T, dv))
    a, b = np.full(T, 0.9), np.full(T, 0.5)
    M0 = rng.standard_normal((N, dv))
    out = O.forward_slice(M0, Pq, Pk, q, kk, v, a, b, N, k, k, "f64")
    iw, _, ww = O.address(Pk, kk, N, k)
    ir, _, wr = O.address(Pq, q, N, k)
    M_ref, y_ref = _dense_masked_sdm(M0, iw, ww, ir, wr, v, a, b)
    np.testing.assert_allclose(out["y64"], y_ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(out["M"], M_ref, rtol=1e-12, atol=1e-12)
    assert np.array_equal(M0, O.forward_slice(M0, Pq, Pk, q, kk, v, a, b, N, k, k, "f64")["M"]) is False


# ------------------------------------------------------------------ chunkwise (WY) form

def _brute_sparse_ip(ia, va, la, ib, vb, lb):
    return sum(va[n] * vb[m] * math.exp(la[n] - lb[m]) for n in range(len(ia)) for m in range(len(ib)) if ia[n] == ib[m])


def test_sparse_ip_two_pointer_equals_brute_force():
    rng = np.random.default_rng(41)
    for _ in range(200):
        ka, kb = rng.integers(1, 9, 2)
        ia = np.sort(rng.choice(20, ka, replace=False))
        ib = np.sort(rng.choice(20, kb, replace=False))
        va, vb = rng.standard_normal(ka), rng.standard_normal(kb)
        la, lb = -rng.uniform(0, 3, ka), -rng.uniform(0, 3, kb)
        assert abs(O.sparse_ip(ia, va, la, ib, vb, lb) - _brute_sparse_ip(ia, va, la, ib, vb, lb)) < 1e-13


@pytest.mark.parametrize("C", [1, 3, 8, 60])
@pytest.mark.parametrize("N", [40, 9])          # N = 9 with 5 writes per token: slots collide constantly
def test_chunkwise_equals_dense_masked_form(C, N):
    rng = np.random.default_rng(42 + N)
    M0, idx_w, w_w, idx_r, w_r, V, alpha, beta = _random_sparse_case(rng, N=N, T=60)
    M = M0.copy()
    y64, _ = O.recur_chunkwise(M, idx_w, w_w, idx_r, w_r, V, alpha, beta, C, "f64")
    M_ref, y_ref = _dense_masked_sdm(M0, idx_w, w_w, idx_r, w_r, V, alpha, beta)
    np.testing.assert_allclose(y64, y_ref, rtol=1e-11, atol=1e-11)
    np.testing.assert_allclose(M, M_ref, rtol=1e-11, atol=1e-11)


def test_chunkwise_gdn_special_case():
    """All slots selected with dense key weights (Sec. 3.1 "Connection to GDN"): the chunkwise form
    is the chunkwise GDN, and equals the textbook GDN update token by token."""
    rng = np.random.default_rng(43)
    dqk, dv, T = 6, 5, 24
    M0 = rng.standard_normal((dqk, dv))
    K = rng.standard_normal((T, dqk)) / np.sqrt(dqk)
    Q = rng.standard_normal((T, dqk))
    V = rng.standard_normal((T, dv))
    a = rng.uniform(0.7, 1.0, T)
    b = rng.uniform(0.1, 0.9, T)
    alls = np.tile(np.arange(dqk), (T, 1))
    M = M0.copy()
    y64, _ = O.recur_chunkwise(M, alls, K, alls, Q, V, a, b, 8, "f64")
    M_ref, y_ref = _gdn_textbook(M0, K, V, Q, a, b)
    np.testing.assert_allclose(y64, y_ref, rtol=1e-11, atol=1e-11)
    np.testing.assert_allclose(M, M_ref, rtol=1e-11, atol=1e-11)


def test_chunkwise_rounding_only_at_chunk_boundaries():
    """With bf16 storage the chunkwise form rounds the memory at chunk boundaries only, and its reads
    within a chunk see the unrounded intra-chunk writes (the token-serial form reads rows rounded
    after each token).  So the two forms differ by bf16 rounding alone, for any C."""
    rng = np.random.default_rng(44)
    M0, idx_w, w_w, idx_r, w_r, V, alpha, beta = _random_sparse_case(rng, N=50, T=48)
    M0 = O.round_storage(M0 * 0.02, "bf16")
    V = O.round_storage(V, "bf16")
    Ms = M0.copy()
    _, ys = O.recur(Ms, idx_w, w_w, idx_r, w_r, V, alpha, beta, "bf16")
    Me = M0.copy()
    ye, _ = O.recur(Me, idx_w, w_w, idx_r, w_r, V, alpha, beta, "f64")    # exact storage
    rel = lambda a, b: np.linalg.norm(a - b) / np.linalg.norm(b)
    # a read row has gone through at most max_writes roundings (2^-9 relative each) plus its own
    bound = (1 + np.bincount(idx_w.ravel()).max()) * 2.0 ** -9
    assert rel(ys, ye) < bound
    for C in (1, 8, 48):
        Mc = M0.copy()
        _, yc = O.recur_chunkwise(Mc, idx_w, w_w, idx_r, w_r, V, alpha, beta, C, "bf16")
        assert rel(yc, ye) < bound, C
        assert np.array_equal(O.round_storage(Mc, "bf16"), Mc)              # stored rows are bf16 values
        touched = np.unique(idx_w)
        assert rel(Mc[touched], Me[touched]) < bound, C


# ------------------------------------------------------------------ backward with in-place undo

def _torch_dense_loss(M0, idx_w, w_w, idx_r, w_r, V, alpha, beta, dy):
    """sum_t <dy_t, y_t> of the dense masked update written in torch (autograd does the rest)."""
    import torch
    N = M0.shape[0]
    M = M0
    loss = 0.0
    for t in range(V.shape[0]):
        mask = torch.zeros(N, dtype=torch.float64).index_put((torch.as_tensor(idx_w[t]),), torch.ones(len(idx_w[t]), dtype=torch.float64))
        kappa = torch.zeros(N, dtype=torch.float64).index_put((torch.as_tensor(idx_w[t]),), w_w[t])
        rho = torch.zeros(N, dtype=torch.float64).index_put((torch.as_tensor(idx_r[t]),), w_r[t])
        Mt = (1.0 + (alpha[t] - 1.0) * mask)[:, None] * M
        M = Mt + beta[t] * torch.outer(kappa, V[t] - Mt.T @ kappa)
        loss = loss + dy[t] @ (M.T @ rho)
    return loss


@pytest.mark.parametrize("N", [30, 7])
def test_backward_with_undo_equals_autograd_of_the_dense_form(N):
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(61 + N)
    M0, idx_w, w_w, idx_r, w_r, V, alpha, beta = _random_sparse_case(rng, N=N, T=25, kw=4, kr=3)
    dy = rng.standard_normal(V.shape)
    M = M0.copy()
    y, undo = O.recur_forward_undo(M, idx_w, w_w, idx_r, w_r, V, alpha, beta)
    M_ref, y_ref = _dense_masked_sdm(M0, idx_w, w_w, idx_r, w_r, V, alpha, beta)
    np.testing.assert_allclose(y, y_ref, rtol=1e-12, atol=1e-12)
    g = O.recur_backward(M, undo, idx_w, w_w, idx_r, w_r, V, alpha, beta, dy)
    assert np.array_equal(M, M0)                                   # the undo restored M_0 exactly
    leaf = lambda a: torch.tensor(a, dtype=torch.float64, requires_grad=True)
    tM0, tww, twr, tV, ta, tb = map(leaf, (M0, w_w, w_r, V, alpha, beta))
    loss = _torch_dense_loss(tM0, idx_w, tww, idx_r, twr, tV, ta, tb, torch.tensor(dy))
    loss.backward()
    for name, t in (("dM0", tM0), ("dw_w", tww), ("dw_r", twr), ("dv", tV), ("dalpha", ta), ("dbeta", tb)):
        np.testing.assert_allclose(g[name], t.grad.numpy(), rtol=1e-10, atol=1e-11, err_msg=name)


def test_backward_finite_differences():
    rng = np.random.default_rng(63)
    M0, idx_w, w_w, idx_r, w_r, V, alpha, beta = _random_sparse_case(rng, N=12, T=10, kw=3, kr=3)
    dy = rng.standard_normal(V.shape)
    def loss(a=alpha, b=beta, vv=V, m0=M0):
        M = m0.copy()
        y, _ = O.recur_forward_undo(M, idx_w, w_w, idx_r, w_r, vv, a, b)
        return float(np.sum(dy * y))
    M = M0.copy()
    _, undo = O.recur_forward_undo(M, idx_w, w_w, idx_r, w_r, V, alpha, beta)
    g = O.recur_backward(M, undo, idx_w, w_w, idx_r, w_r, V, alpha, beta, dy)
    h = 1e-6
    for t in (0, 4, 9):
        e = np.zeros_like(alpha)
        e[t] = h
        assert abs((loss(a=alpha + e) - loss(a=alpha - e)) / (2 * h) - g["dalpha"][t]) < 1e-7
        assert abs((loss(b=beta + e) - loss(b=beta - e)) / (2 * h) - g["dbeta"][t]) < 1e-7
    i = int(idx_w[2, 1])
    E = np.zeros_like(M0)
    E[i, 0] = h
    assert abs((loss(m0=M0 + E) - loss(m0=M0 - E)) / (2 * h) - g["dM0"][i, 0]) < 1e-7


def test_e4m3_rounding_equals_torch_float8():
    torch = pytest.importorskip("torch")
    if not hasattr(torch, "float8_e4m3fn"):
        pytest.skip("torch without float8")
    rng = np.random.default_rng(64)
    x = np.concatenate([rng.standard_normal(4000) * 10.0 ** rng.integers(-4, 3, 4000),
                        [0.0, 448.0, -448.0, 2.0 ** -6, 2.0 ** -9, 2.0 ** -10, 1.0625, 1.1875, 3 * 2.0 ** -10]])
    x = np.clip(x, -448.0, 448.0).astype(np.float32).astype(np.float64)
    ref = torch.from_numpy(x.astype(np.float32)).to(torch.float8_e4m3fn).to(torch.float64).numpy()
    assert np.array_equal(O.round_e4m3(x), ref)


def test_quantized_undo_log_bounds_and_effect_on_gradients():
    """A quantised snapshot (App. A.3) restores each logged row within half a quantisation step
    (fp8: 2^-4 relative to the row's largest entry at worst; int4: max|row| / 14); the backward
    then restores an approximate M_0, and its gradients move further from the exact ones for the
    coarser format."""
    rng = np.random.default_rng(65)
    M0, idx_w, w_w, idx_r, w_r, V, alpha, beta = _random_sparse_case(rng, N=30, T=40, kw=4, kr=3)
    dy = rng.standard_normal(V.shape)
    M = M0.copy()
    _, undo = O.recur_forward_undo(M, idx_w, w_w, idx_r, w_r, V, alpha, beta)
    amax = np.max(np.abs(undo), axis=-1, keepdims=True)
    assert np.all(np.abs(O.quantize_undo(undo, "fp8") - undo) <= amax * 2.0 ** -4 + 1e-300)
    assert np.all(np.abs(O.quantize_undo(undo, "int4") - undo) <= amax / 14 * (1 + 1e-12))
    assert np.array_equal(O.quantize_undo(undo, "exact"), undo)
    ref = O.recur_backward(M.copy(), undo, idx_w, w_w, idx_r, w_r, V, alpha, beta, dy)
    err = {}
    for kind in ("fp8", "int4"):
        g = O.recur_backward(M.copy(), O.quantize_undo(undo, kind), idx_w, w_w, idx_r, w_r, V, alpha, beta, dy)
        err[kind] = max(np.linalg.norm(g[n] - ref[n]) / np.linalg.norm(ref[n]) for n in ("dv", "dalpha", "dw_w", "dM0"))
    assert 0 < err["fp8"] < err["int4"] and err["fp8"] < 0.1


def test_undo_codes_in_float32_arithmetic():
    """The snapshot codes as a float32 implementation decides them: hand-worked int4 row with
    ties to even, the row maximum always coded as the top value, codes inside the format, the
    float64 path reproduced exactly where the scale is a power of two (every step exact), and
    the half-step error bound of the float32 dequantised rows."""
    # s = 7 / 7 = 1: codes are the integers nearest the entries, ties to even
    row = np.array([[7.0, 3.5, -3.5, 0.5, 1.5, 2.5, -6.5, 0.0]])
    q, sc = O.undo_codes(row, "int4")
    assert sc.tolist() == [1.0]
    assert q.tolist() == [[7, 4, -4, 0, 2, 2, -6, 0]]
    # fp8: max 448 -> s = 1; 1.0625 lies halfway between 1 and 1.125 (4 significant bits): to even
    row = np.array([[448.0, 1.0625, 1.1875, -2.0 ** -9, 3.0 * 2.0 ** -10, 0.0]])
    q, sc = O.undo_codes(row, "fp8")
    assert sc.tolist() == [1.0]
    assert q.tolist() == [[448.0, 1.0, 1.25, -2.0 ** -9, 2.0 ** -8, 0.0]]
    # zero rows: scale 1, codes 0
    q, sc = O.undo_codes(np.zeros((2, 5)), "fp8")
    assert sc.tolist() == [1.0, 1.0] and not q.any()
    rng = np.random.default_rng(66)
    u = (rng.standard_normal((40, 9, 32)) * np.exp(3 * rng.standard_normal((40, 9, 1)))).astype(np.float32)
    u = u.astype(np.float64)
    for kind, top in (("fp8", 448.0), ("int4", 7.0)):
        q, sc = O.undo_codes(u, kind)
        assert sc.dtype == np.float32
        amax = np.abs(u).max(axis=-1)
        assert np.all(np.abs(q).max(axis=-1) == top)                     # the row maximum codes as +-top
        if kind == "int4":
            assert np.array_equal(q, np.round(q)) and np.abs(q).max() <= 7
        else:
            assert np.array_equal(O.round_e4m3(q), q)
        deq = O.quantize_undo(u, kind, "f32")
        step = amax * (2.0 ** -4 if kind == "fp8" else 1.0 / 14.0)
        assert np.all(np.abs(deq - u) <= step[..., None] * (1 + 2.0 ** -20) + 1e-300)
        # rows scaled so that max|row| = top * 2^e: the scale is a power of two, every step exact
        p2 = (u / amax[..., None] * top).astype(np.float32).astype(np.float64)
        p2 = p2 * 2.0 ** rng.integers(-8, 8, amax.shape)[..., None]
        assert np.array_equal(O.quantize_undo(p2, kind, "f32"), O.quantize_undo(p2, kind))


# ------------------------------------------------------------------ lazy M0 (copy-on-write)

def test_lazy_overlay_equals_dense_masked_form():
    """The copy-on-write memory (overlay of written rows over a read-only M0) gives the
    dense update's y and final memory; its keys are exactly the slots ever written."""
    rng = np.random.default_rng(21)
    M0, idx_w, w_w, idx_r, w_r, V, alpha, beta = _random_sparse_case(rng, N=60, T=70)
    M0_ro = M0.copy()
    M0_ro.setflags(write=False)
    overlay = {}
    y64, _ = O.recur_lazy(M0_ro, overlay, idx_w, w_w, idx_r, w_r, V, alpha, beta, "f64")
    M_ref, y_ref = _dense_masked_sdm(M0, idx_w, w_w, idx_r, w_r, V, alpha, beta)
    np.testing.assert_allclose(y64, y_ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(O.materialize(M0_ro, overlay), M_ref, rtol=1e-12, atol=1e-12)
    written = set(int(s) for s in idx_w.ravel())
    assert set(overlay) == written
    mask = O.touched_mask(idx_w, M0.shape[0])
    assert np.array_equal(np.flatnonzero(mask), np.array(sorted(written)))
    # slots never written keep M0 exactly
    assert np.array_equal(O.materialize(M0_ro, overlay)[~mask], M0[~mask])


def test_lazy_continuation_and_prior_mask():
    """A sequence split over two calls carries the overlay (and the touched mask with it)."""
    rng = np.random.default_rng(22)
    M0, idx_w, w_w, idx_r, w_r, V, alpha, beta = _random_sparse_case(rng, N=50, T=64)
    M0 = O.round_storage(M0 * 0.02, "bf16")
    V = O.round_storage(V, "bf16")
    ov_a = {}
    _, ya = O.recur_lazy(M0, ov_a, idx_w, w_w, idx_r, w_r, V, alpha, beta, "bf16")
    ov_b = {}
    c = 29
    _, yb1 = O.recur_lazy(M0, ov_b, idx_w[:c], w_w[:c], idx_r[:c], w_r[:c], V[:c], alpha[:c], beta[:c], "bf16")
    m1 = O.touched_mask(idx_w[:c], 50)
    _, yb2 = O.recur_lazy(M0, ov_b, idx_w[c:], w_w[c:], idx_r[c:], w_r[c:], V[c:], alpha[c:], beta[c:], "bf16")
    assert np.array_equal(ya, np.concatenate([yb1, yb2]))
    assert set(ov_a) == set(ov_b) and all(np.array_equal(ov_a[s], ov_b[s]) for s in ov_a)
    assert np.array_equal(O.touched_mask(idx_w[c:], 50, prior=m1), O.touched_mask(idx_w, 50))
    Md = M0.copy()
    _, yd = O.recur(Md, idx_w, w_w, idx_r, w_r, V, alpha, beta, "bf16")
    assert np.array_equal(yd, ya) and np.array_equal(O.materialize(M0, ov_a), Md)


# ------------------------------------------------------------------ access diagnostics

@pytest.mark.parametrize("k", [1, 4, 32, 64])
def test_eff_keys_and_cumulative_mass_closed_forms(k):
    uniform = np.full((3, k), 1.0 / k)
    np.testing.assert_allclose(O.eff_keys_fraction(uniform), 1.0, rtol=1e-14)
    np.testing.assert_allclose(O.cumulative_mass(uniform), np.tile(np.arange(1, k + 1) / k, (3, 1)), rtol=1e-14)
    onehot = np.zeros((2, k))
    onehot[0, k - 1] = 1.0
    onehot[1, 0] = 1.0
    np.testing.assert_allclose(O.eff_keys_fraction(onehot), 1.0 / k, rtol=1e-14)
    np.testing.assert_allclose(O.cumulative_mass(onehot), 1.0, rtol=1e-14)
    if k >= 2:
        # mass split evenly over two keys: exp(H) = 2, C = [1/2, 1, 1, ...]
        two = np.zeros(k)
        two[[0, k - 1]] = 0.5
        np.testing.assert_allclose(O.eff_keys_fraction(two), 2.0 / k, rtol=1e-14)
        np.testing.assert_allclose(O.cumulative_mass(two), np.r_[0.5, np.ones(k - 1)], rtol=1e-14)
        # geometric weights p_i = (1-r) r^i / (1 - r^k): H in closed form
        r = 0.7
        i = np.arange(k)
        p = (1 - r) * r ** i / (1 - r ** k)
        H = -np.sum(p * (np.log((1 - r) / (1 - r ** k)) + i * np.log(r)))
        rng = np.random.default_rng(23)
        pp = rng.permutation(p)
        np.testing.assert_allclose(O.eff_keys_fraction(pp), np.exp(H) / k, rtol=1e-12)
        np.testing.assert_allclose(O.cumulative_mass(pp), (1 - r ** (i + 1)) / (1 - r ** k), rtol=1e-12)


def test_cumulative_mass_invariants_on_softmax_weights():
    rng = np.random.default_rng(24)
    z = rng.standard_normal((50, 16)) * 2
    p = np.exp(z) / np.exp(z).sum(axis=1, keepdims=True)
    C = O.cumulative_mass(p)
    np.testing.assert_allclose(C[:, -1], 1.0, rtol=1e-13)
    assert np.all(np.diff(C, axis=1) >= 0) and np.all(np.diff(C, n=2, axis=1) <= 1e-15)   # nondecreasing, concave
    np.testing.assert_allclose(C[:, 0], p.max(axis=1), rtol=1e-15)
    u = O.eff_keys_fraction(p)
    assert np.all(u > 1.0 / 16 - 1e-15) and np.all(u <= 1.0 + 1e-15)


def test_unique_fraction_counts():
    N = 64
    # literal count: slots {3, 5, 9, 60} appear (with repeats), so 4 of 64 are unique
    assert O.unique_fraction(np.array([[3, 5, 9], [5, 9, 60], [3, 3, 60]]), N) == 4 / 64
    assert O.unique_fraction(np.arange(N).reshape(8, 8), N) == 1.0
    assert O.unique_fraction(np.full((5, 3), 7), N) == 1.0 / N
    rng = np.random.default_rng(25)
    idx = rng.integers(0, N, (40, 4))
    assert O.unique_fraction(idx, N) == len(set(idx.ravel().tolist())) / N


# ------------------------------------------------------------------ gates and output epilogue

def test_softplus_known_values_and_asymptotes():
    np.testing.assert_allclose(O.softplus(np.array([0.0])), [math.log(2.0)], rtol=1e-15)
    z = np.array([-800.0, -30.0, 30.0, 800.0])
    np.testing.assert_allclose(O.softplus(z), [0.0, math.exp(-30.0), 30.0 + math.exp(-30.0), 800.0], rtol=1e-12)
    zz = np.linspace(-5, 5, 41)
    np.testing.assert_allclose(O.softplus(zz) - O.softplus(-zz), zz, atol=1e-14)   # softplus(z) - softplus(-z) = z


def test_gates_closed_forms():
    """W = 0: alpha = exp(-A c) when b_dt = inv_softplus(c), beta = 1/2; A = 0: alpha = 1;
    beta(-z) = 1 - beta(z); the paper's initialisation keeps softplus(b_dt) in [0.001, 0.1]."""
    rng = np.random.default_rng(31)
    T, d, H = 7, 12, 5
    x = rng.standard_normal((T, d))
    c = rng.uniform(0.001, 0.1, H)
    b_dt = np.log(np.expm1(c))
    A = rng.uniform(0, 16, H)
    alpha, beta = O.gates(x, np.zeros((H, d)), b_dt, A, np.zeros((H, d)))
    np.testing.assert_allclose(alpha, np.tile(np.exp(-A * c)[:, None], (1, T)), rtol=1e-13)
    np.testing.assert_allclose(beta, 0.5, rtol=1e-15)
    W = rng.standard_normal((H, d))
    a1, b1 = O.gates(x, W, b_dt, np.zeros(H), W)
    a2, b2 = O.gates(-x, W, b_dt, np.zeros(H), W)
    np.testing.assert_allclose(a1, 1.0, rtol=1e-15)
    np.testing.assert_allclose(b1 + b2, 1.0, rtol=1e-14)
    # one explicit token and head, summed by hand
    za = sum(W[2, i] * x[3, i] for i in range(d)) + b_dt[2]
    al, _ = O.gates(x, W, b_dt, A, W)
    np.testing.assert_allclose(al[2, 3], math.exp(-A[2] * math.log1p(math.exp(za))), rtol=1e-13)


def test_norm_gate_closed_forms_and_invariance():
    rng = np.random.default_rng(32)
    T, dv = 6, 16
    g = rng.uniform(0, 1, (T, dv))
    gamma = 1 + 0.1 * rng.standard_normal(dv)
    c = rng.uniform(0.5, 3, T) * rng.choice([-1, 1], T)
    y = np.tile(c[:, None], (1, dv))                     # constant rows: RMSNorm(y) = sign(c)
    np.testing.assert_allclose(O.norm_gate(y, g, gamma, 0.0), g * gamma[None, :] * np.sign(c)[:, None], rtol=1e-14)
    y = rng.standard_normal((T, dv))
    s = rng.uniform(0.1, 10, T)[:, None]
    np.testing.assert_allclose(O.norm_gate(s * y, g, gamma, 0.0), O.norm_gate(y, g, gamma, 0.0), rtol=1e-13)
    z = O.norm_gate(y, np.ones((T, dv)), np.ones(dv), 0.0)
    np.testing.assert_allclose(np.mean(z * z, axis=1), 1.0, rtol=1e-13)   # unit mean square
    # eps: rows of zeros stay zero, and eps > 0 shrinks the norm
    assert np.all(O.norm_gate(np.zeros((2, dv)), g[:2], gamma, 1e-6) == 0)
    assert np.all(np.abs(O.norm_gate(y, g, gamma, 1e-2)) < np.abs(O.norm_gate(y, g, gamma, 0.0)))


def test_head_mix_two_heads_by_hand():
    """Two heads, one token, d_v = 2, d = 2, worked by hand: concat(z_0, z_1) = [1, 2, 3, 4];
    W_o rows [1, 0, 0, 1] and [0, 1, -1, 0] give o = [1 + 4, 2 - 3] = [5, -1]; the heads
    concatenated in the wrong order would give [5, 3]."""
    z = np.array([[[1.0, 2.0]], [[3.0, 4.0]]])            # [H=2, T=1, d_v=2]
    W = np.array([[1.0, 0.0, 0.0, 1.0], [0.0, 1.0, -1.0, 0.0]])
    assert np.array_equal(O.head_mix(z, W), np.array([[5.0, -1.0]]))


def test_head_mix_is_a_sum_over_heads():
    rng = np.random.default_rng(33)
    H, T, dv, d = 3, 4, 5, 7
    z = rng.standard_normal((H, T, dv))
    W = rng.standard_normal((d, H * dv))
    o = O.head_mix(z, W)
    ref = sum(z[h] @ W[:, h * dv:(h + 1) * dv].T for h in range(H))
    np.testing.assert_allclose(o, ref, rtol=1e-13, atol=1e-13)


# ------------------------------------------------------------------ geometry (printed numbers)

def test_table1_sdm_state_sizes():
    for level, d, layers, H, printed in _golden_rows("table1_sdm_state.txt"):
        d, layers, H, printed = int(d), int(layers), int(H), float(printed)
        total = O.n_global_layers(layers) * O.state_elements_per_layer(d, H)
        digits = 4 if printed >= 1e9 else (3 if printed >= 1e8 else 2)
        assert float(f"{total:.{digits}g}") == printed, (level, total, printed)


def test_table3_state_per_layer_mb():
    for d, H, dqk, printed in _golden_rows("table3_state_per_layer.txt"):
        d, H, dqk, printed = int(d), int(H), int(dqk), int(printed)
        n = (dqk // (2 * H)) ** 2                # per-head key = 2 sqrt(N), d_qk per head = dqk / H
        mib = H * n * (d // H) * 2 / 2 ** 20
        assert round(mib) == printed, (d, H, dqk, mib)
    assert O.state_elements_per_layer(1920, 2) * 2 / 2 ** 20 == pytest.approx(211, abs=0.5)


def test_appendix_a3_checkpoint_sizes():
    printed = {name: float(v) for name, v in _golden_rows("appA3_checkpoints.txt")}
    d, H, T, C, W = 3840, 2, 16384, 128, 64
    per_layer = O.state_elements_per_layer(d, H)
    assert round((T // C) * per_layer * 2 / 1e9) == printed["chunk_snapshots"]
    assert round(T * W * d * 2 / 1e9) == printed["undo_log"]


# ------------------------------------------------------------------ planted mistakes

def _recur_per_slot_delta(M, idx_w, w_w, idx_r, w_r, v, alpha, beta):
    # Literal per-slot reading of Eq. sdm-write: v_t - M~_t[i] instead of v_t - v~_t.
    ys = []
    for t in range(v.shape[0]):
        d = alpha[t] * M[idx_w[t]]
        M[idx_w[t]] = d + beta[t] * w_w[t][:, None] * (v[t][None, :] - d)
        ys.append(w_r[t] @ M[idx_r[t]])
    return np.array(ys)


def _recur_read_before_write(M, idx_w, w_w, idx_r, w_r, v, alpha, beta):
    ys = []
    for t in range(v.shape[0]):
        ys.append(w_r[t] @ M[idx_r[t]])
        d = alpha[t] * M[idx_w[t]]
        M[idx_w[t]] = d + beta[t] * w_w[t][:, None] * (v[t] - w_w[t] @ d)[None, :]
    return np.array(ys)


def _recur_global_decay(M, idx_w, w_w, idx_r, w_r, v, alpha, beta):
    ys = []
    for t in range(v.shape[0]):
        M *= alpha[t]
        d = M[idx_w[t]]
        M[idx_w[t]] = d + beta[t] * w_w[t][:, None] * (v[t] - w_w[t] @ d)[None, :]
        ys.append(w_r[t] @ M[idx_r[t]])
    return np.array(ys)


def test_pins_reject_planted_mistakes():
    rng = np.random.default_rng(17)
    dqk, dv, T = 6, 5, 30
    M0 = rng.standard_normal((dqk, dv))
    K = rng.standard_normal((T, dqk)) / np.sqrt(dqk)
    Q = rng.standard_normal((T, dqk))
    V = rng.standard_normal((T, dv))
    a = np.full(T, 0.9)
    b = np.full(T, 0.7)
    alls = np.tile(np.arange(dqk), (T, 1))
    _, y_gdn = _gdn_textbook(M0, K, V, Q, a, b)
    assert not np.allclose(_recur_per_slot_delta(M0.copy(), alls, K, alls, Q, V, a, b), y_gdn, atol=1e-6)
    assert not np.allclose(_recur_read_before_write(M0.copy(), alls, K, alls, Q, V, a, b), y_gdn, atol=1e-6)
    M0s, iw, ww, ir, wr, Vs, al, _ = _random_sparse_case(rng)
    M = M0s.copy()
    _recur_global_decay(M, iw, ww, ir, wr, Vs, al, np.zeros(Vs.shape[0]))
    decay = np.ones(M0s.shape[0])
    for t in range(Vs.shape[0]):
        decay[iw[t]] *= al[t]
    assert not np.allclose(M, decay[:, None] * M0s)
    # a transposed outer-sum flattening (slot = j*S + i) fails the brute-force pin
    s1, s2 = rng.standard_normal(8), rng.standard_normal(8)
    idx, _, _ = O.pkm_select(s2[None], s1[None], 4)
    assert not np.array_equal(idx[0], _brute_topk(s1, s2, 4))
    # a copy-on-write memory whose reads ignore the overlay (always M0) fails the dense pin
    M0c, iw, ww, ir, wr, Vc, al, be = _random_sparse_case(rng)
    _, y_ref = _dense_masked_sdm(M0c, iw, ww, ir, wr, Vc, al, be)
    ys = []
    ov = {}
    for t in range(Vc.shape[0]):
        d = [al[t] * (ov[s] if s in ov else M0c[s]) for s in iw[t]]
        pred = sum(ww[t][n] * d[n] for n in range(len(d)))
        for n, s in enumerate(iw[t]):
            ov[s] = d[n] + be[t] * ww[t][n] * (Vc[t] - pred)
        ys.append(sum(wr[t][n] * M0c[s] for n, s in enumerate(ir[t])))
    assert not np.allclose(np.array(ys), y_ref, atol=1e-6)
    # effective keys without the exponential (entropy / k) fails the two-key closed form
    two = np.array([0.5, 0.0, 0.0, 0.5])
    assert not np.isclose(-np.sum(np.where(two > 0, two * np.log(np.where(two > 0, two, 1)), 0)) / 4, 2.0 / 4)
    # cumulative mass of the weights in slot order (unsorted) fails the geometric closed form
    p = np.array([0.1, 0.6, 0.3])
    assert not np.allclose(np.cumsum(p), O.cumulative_mass(p))
    # chunkwise form without the decay factor in A, or with beta of the column token in M_sys,
    # fails the dense pin
    M0w, iw, ww, ir, wr, Vw, al, be = _random_sparse_case(rng, N=9, T=20)
    _, y_ref = _dense_masked_sdm(M0w, iw, ww, ir, wr, Vw, al, be)
    def chunk_variant(no_decay_in_A=False, beta_col=False):
        n = Vw.shape[0]
        acc, lw, lr = {}, np.zeros(iw.shape), np.zeros(ir.shape)
        for t in range(n):
            for m, i in enumerate(iw[t]):
                acc[int(i)] = acc.get(int(i), 0.0) + math.log(al[t])
                lw[t, m] = acc[int(i)]
            for m, j in enumerate(ir[t]):
                lr[t, m] = acc.get(int(j), 0.0)
        z = lambda x: np.zeros_like(x) if no_decay_in_A else x
        A = np.array([[O.sparse_ip(iw[t], ww[t], z(lw[t]), iw[s_], ww[s_], z(lw[s_])) if s_ < t else 0.0
                       for s_ in range(n)] for t in range(n)])
        QK = np.array([[O.sparse_ip(ir[t], wr[t], lr[t], iw[s_], ww[s_], lw[s_]) if s_ <= t else 0.0
                        for s_ in range(n)] for t in range(n)])
        Msys = np.eye(n) + (A * be[None, :] if beta_col else be[:, None] * A)
        Minv = np.linalg.inv(Msys)
        ret = np.stack([(ww[t] * np.exp(lw[t])) @ M0w[iw[t]] for t in range(n)])
        inter = np.stack([(wr[t] * np.exp(lr[t])) @ M0w[ir[t]] for t in range(n)])
        u = Minv @ (be[:, None] * Vw) - Minv @ (be[:, None] * ret)
        return inter + QK @ u
    assert np.allclose(chunk_variant(), y_ref, atol=1e-10)             # the variant machinery is right
    assert not np.allclose(chunk_variant(no_decay_in_A=True), y_ref, atol=1e-6)
    assert not np.allclose(chunk_variant(beta_col=True), y_ref, atol=1e-6)
    # a backward that reads the pre-write memory (the read-before-write mistake) fails autograd
    torch_mod = pytest.importorskip("torch")
    M0b, iwb, wwb, irb, wrb, Vb, alb, beb = _random_sparse_case(rng, N=7, T=12, kw=4, kr=3)
    dyb = rng.standard_normal(Vb.shape)
    Mb = M0b.copy()
    _, und = O.recur_forward_undo(Mb, iwb, wwb, irb, wrb, Vb, alb, beb)
    gb = O.recur_backward(Mb, und, iwb, wwb, irb, wrb, Vb, alb, beb, dyb)
    lf = lambda a: torch_mod.tensor(a, dtype=torch_mod.float64, requires_grad=True)
    tw = lf(wrb)
    _torch_dense_loss(torch_mod.tensor(M0b), iwb, torch_mod.tensor(wwb), irb, tw, torch_mod.tensor(Vb),
                      torch_mod.tensor(alb), torch_mod.tensor(beb), torch_mod.tensor(dyb)).backward()
    np.testing.assert_allclose(gb["dw_r"], tw.grad.numpy(), rtol=1e-10, atol=1e-11)
    Mw = M0b.copy()
    wrong = np.zeros(wrb.shape)
    for t in range(Vb.shape[0]):                                 # d rho from M_{t-1} instead of M_t
        wrong[t] = Mw[irb[t]] @ dyb[t]
        d_ = alb[t] * Mw[iwb[t]]
        Mw[iwb[t]] = d_ + beb[t] * wwb[t][:, None] * (Vb[t] - wwb[t] @ d_)[None, :]
    assert not np.allclose(wrong, tw.grad.numpy(), atol=1e-6)
    # RMSNorm without the square root (y / mean(y^2)) fails the scale invariance
    y = rng.standard_normal((3, 8))
    bad = lambda yy: yy / np.mean(yy * yy, axis=-1, keepdims=True)
    assert not np.allclose(bad(4.0 * y), bad(y))
    # softplus replaced by max(z, 0) fails softplus(0) = log 2
    assert not np.isclose(max(0.0, 0.0), math.log(2.0))
    # a gate without the bias fails the W = 0 closed form
    c = np.array([0.05])
    assert not np.isclose(np.exp(-3.0 * O.softplus(0.0)), np.exp(-3.0 * c[0]))
