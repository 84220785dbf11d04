"""Pins for the fp64 oracle against what the paper and the mathematics fix.

Each test checks the sequential learner in ``oracle/`` against something other
than itself: the closed form of Eq. 2, the dense scan-read identity of
Appendix C, plain GEMMs in the degenerate cases, linearity, Theorem 1
recovery from an independently written serial learner, the Sec. 4.1
experiment, and finite differences for the activation derivatives.
"""
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rng(seed):
    return np.random.default_rng(seed)


def _rand_problem(seed, U, T, d, m, scale_g=1.0):
    r = _rng(seed)
    x = r.standard_normal((U, T, d)) / np.sqrt(d)
    ghat = r.standard_normal((U, T, m)) * scale_g
    W0 = r.standard_normal((U, m, d)) / np.sqrt(d)
    gout = r.standard_normal((U, T, m))
    return x, ghat, W0, gout


# --------------------------------------------------------------------------- Eq. 2
def _closed_form_delta(t, x, g, eta, alpha):
    """Delta_t = -sum_{i<t} eta_i (prod_{j=i+1}^{t-1} alpha_j) g_i x_i^T (Eq. 2),
    with empty sums zero and empty products one."""
    m, d = g.shape[1], x.shape[1]
    D = np.zeros((m, d))
    for i in range(t):
        prod = 1.0
        for j in range(i + 1, t):
            prod *= alpha[j]
        D -= eta[i] * prod * np.outer(g[i], x[i])
    return D


@pytest.mark.parametrize("T,d,m", [(1, 3, 2), (2, 4, 3), (5, 3, 4), (8, 6, 5)])
def test_closed_form_eq2_with_gates(T, d, m):
    x, ghat, W0, gout = _rand_problem(100 + T, 1, T, d, m)
    r = _rng(7 + T)
    eta = r.uniform(0.05, 0.5, T)
    alpha = r.uniform(0.3, 1.0, T)
    y, gin = oracle.linear_scan(x, ghat, W0, eta, alpha=alpha, gout=gout)
    for t in range(T):
        W_t = W0[0] + _closed_form_delta(t, x[0], ghat[0], eta, alpha)
        np.testing.assert_allclose(y[0, t], W_t @ x[0, t], rtol=0, atol=1e-14)
        np.testing.assert_allclose(gin[0, t], W_t.T @ gout[0, t], rtol=0, atol=1e-14)


@pytest.mark.parametrize("T", [6, 11])
def test_closed_form_eq2_resets_and_negative_retention(T):
    """alpha_t = 0 (resets, also two in a row) and alpha_t < 0 still follow Eq. 2."""
    x, ghat, W0, gout = _rand_problem(300 + T, 1, T, 5, 4)
    r = _rng(8 + T)
    eta = r.uniform(0.05, 0.5, T)
    alpha = r.uniform(0.5, 1.0, T)
    alpha[[1, 3, 4]] = 0.0
    alpha[T - 2] = -0.7
    y, gin = oracle.linear_scan(x, ghat, W0, eta, alpha=alpha, gout=gout)
    for t in range(T):
        W_t = W0[0] + _closed_form_delta(t, x[0], ghat[0], eta, alpha)
        np.testing.assert_allclose(y[0, t], W_t @ x[0, t], rtol=0, atol=1e-14)
        np.testing.assert_allclose(gin[0, t], W_t.T @ gout[0, t], rtol=0, atol=1e-14)


def test_reset_restarts_a_fresh_learner():
    """After alpha_r = 0 the map is W0 minus the writes from token r on, so every read
    after r equals the read of a learner started at token r from W0 (whatever alpha_r)."""
    T, rr = 40, 17
    x, ghat, W0, gout = _rand_problem(77, 1, T, 8, 6)
    r = _rng(78)
    eta = r.uniform(0.05, 0.3, T)
    alpha = r.uniform(0.6, 1.0, T)
    alpha[rr] = 0.0
    y, gin = oracle.linear_scan(x, ghat, W0, eta, alpha=alpha, gout=gout)
    a2 = alpha[rr:].copy()
    a2[0] = 0.37  # scales the fresh learner's zero fast weights: no effect
    y2, g2 = oracle.linear_scan(x[:, rr:], ghat[:, rr:], W0, eta[rr:], alpha=a2, gout=gout[:, rr:])
    # the read at r itself comes before r's write and still sees the history
    np.testing.assert_allclose(y[0, rr + 1:], y2[0, 1:], rtol=0, atol=1e-13)
    np.testing.assert_allclose(gin[0, rr + 1:], g2[0, 1:], rtol=0, atol=1e-13)
    assert np.abs(y[0, rr] - y2[0, 0]).max() > 1e-3


# ---------------------------------------------------- document resets (App. C, E)
def _doc_starts(T, cuts):
    ds = np.zeros((1, T), dtype=bool)
    ds[0, list(cuts)] = True
    return ds


@pytest.mark.parametrize("gated", [False, True])
def test_documents_closed_form(gated):
    """Each read sees W0 plus the writes of its own document only (Appendix C, scan
    reads), checked against the closed form of Eq. 2 over that document's tokens."""
    T, cuts = 13, (1, 5, 6, 10)
    x, ghat, W0, gout = _rand_problem(400 + gated, 1, T, 4, 3)
    r = _rng(401)
    eta = r.uniform(0.05, 0.5, T)
    alpha = r.uniform(0.4, 1.0, T) if gated else np.ones(T)
    y, gin = oracle.linear_scan_docs(x, ghat, W0, eta, _doc_starts(T, cuts),
                                     alpha=alpha if gated else None, gout=gout)
    bounds = [0, *cuts, T]
    for a, b in zip(bounds[:-1], bounds[1:]):
        for t in range(a, b):
            W_t = W0[0] + _closed_form_delta(t - a, x[0, a:b], ghat[0, a:b], eta[a:b], alpha[a:b])
            np.testing.assert_allclose(y[0, t], W_t @ x[0, t], rtol=0, atol=1e-14)
            np.testing.assert_allclose(gin[0, t], W_t.T @ gout[0, t], rtol=0, atol=1e-14)


def test_documents_are_eq2_gates_zeroed_before_each_start():
    """The reading the GPU path takes: a document starting at s is alpha = eta = 0 at
    token s - 1 in the one-sequence recurrence of Eq. 2."""
    T, cuts = 90, (1, 2, 30, 64, 65, 89)
    x, ghat, W0, gout = _rand_problem(402, 1, T, 6, 5)
    r = _rng(403)
    eta = r.uniform(0.02, 0.3, T)
    alpha = r.uniform(0.8, 1.0, T)
    yd, gd = oracle.linear_scan_docs(x, ghat, W0, eta, _doc_starts(T, cuts), alpha=alpha, gout=gout)
    e2, a2 = eta.copy(), alpha.copy()
    for c in cuts:
        e2[c - 1] = 0.0
        a2[c - 1] = 0.0
    y, g = oracle.linear_scan(x, ghat, W0, e2, alpha=a2, gout=gout)
    np.testing.assert_allclose(y, yd, rtol=0, atol=1e-13)
    np.testing.assert_allclose(g, gd, rtol=0, atol=1e-13)


def test_documents_of_one_token_read_slow_weights():
    """Every token its own document: no read sees any write, y_t = W0 x_t."""
    T = 9
    x, ghat, W0, gout = _rand_problem(404, 1, T, 5, 4)
    y, gin = oracle.linear_scan_docs(x, ghat, W0, 0.4, np.ones((1, T), dtype=bool), gout=gout)
    np.testing.assert_allclose(y[0], x[0] @ W0[0].T, rtol=0, atol=1e-14)
    np.testing.assert_allclose(gin[0], gout[0] @ W0[0], rtol=0, atol=1e-14)


def test_first_read_is_slow_weights():
    """W_hat_0 = W_0 (Delta_0 = 0; read before write): row t=0 is a plain GEMV."""
    x, ghat, W0, gout = _rand_problem(3, 4, 6, 16, 8)
    y, gin = oracle.linear_scan(x, ghat, W0, 0.3, gout=gout)
    for u in range(4):
        np.testing.assert_allclose(y[u, 0], W0[u] @ x[u, 0], rtol=0, atol=1e-15)
        np.testing.assert_allclose(gin[u, 0], W0[u].T @ gout[u, 0], rtol=0, atol=1e-15)


# ------------------------------------------------------------ App. C scan reads
def _dense_scan_reads(x, ghat, W0, eta, alpha, gout):
    """Appendix C: Delta_t a_t = -sum_{i<t} eta_i (prod alpha) ghat_i (x_i^T a_t) and
    Delta_t^T b_t = -sum_{i<t} eta_i (prod alpha) x_i (ghat_i^T b_t), written as
    masked products of whole matrices (queries a_t = x_t, b_t = gout_t)."""
    T = x.shape[0]
    la = np.concatenate([[0.0], np.cumsum(np.log(alpha))])  # la[k] = sum_{j<k} log alpha_j
    gamma = np.zeros((T, T))
    for t in range(T):
        for i in range(t):
            # prod_{j=i+1}^{t-1} alpha_j = exp(la[t] - la[i+1])
            gamma[t, i] = eta[i] * np.exp(la[t] - la[i + 1])
    Y = x @ W0.T - (gamma * (x @ x.T)) @ ghat
    G = gout @ W0 - (gamma * (gout @ ghat.T)) @ x
    return Y, G


@pytest.mark.parametrize("T,d,m,gated", [(64, 16, 24, False), (300, 32, 32, False),
                                         (512, 64, 64, False), (200, 12, 20, True)])
def test_dense_scan_read_identity(T, d, m, gated):
    x, ghat, W0, gout = _rand_problem(11 + T, 1, T, d, m)
    r = _rng(T)
    eta = r.uniform(0.01, 0.2, T)
    alpha = r.uniform(0.9, 1.0, T) if gated else np.ones(T)
    y, gin = oracle.linear_scan(x, ghat, W0, eta, alpha=alpha if gated else None, gout=gout)
    Yd, Gd = _dense_scan_reads(x[0], ghat[0], W0[0], eta, alpha, gout[0])
    scale_y = np.abs(Yd).max()
    scale_g = np.abs(Gd).max()
    assert np.abs(y[0] - Yd).max() <= 1e-12 * scale_y
    assert np.abs(gin[0] - Gd).max() <= 1e-12 * scale_g


def test_exclusive_not_inclusive():
    """The read at t excludes the write at t: with one nonzero write at token 3,
    y_3 is still W0 x_3 while y_4 sees the write."""
    T, d, m = 6, 5, 4
    x, ghat, W0, _ = _rand_problem(5, 1, T, d, m)
    g = np.zeros_like(ghat)
    g[0, 3] = ghat[0, 3]
    y, _ = oracle.linear_scan(x, g, W0, 0.7)
    np.testing.assert_allclose(y[0, 3], W0[0] @ x[0, 3], atol=1e-15)
    expect4 = (W0[0] - 0.7 * np.outer(g[0, 3], x[0, 3])) @ x[0, 4]
    np.testing.assert_allclose(y[0, 4], expect4, atol=1e-15)
    assert np.abs(y[0, 4] - W0[0] @ x[0, 4]).max() > 1e-3


# ---------------------------------------------------------- degenerate cases
@pytest.mark.parametrize("which", ["eta0", "ghat0"])
def test_degenerate_is_plain_gemm(which):
    x, ghat, W0, gout = _rand_problem(21, 3, 40, 32, 16)
    eta = 0.0 if which == "eta0" else 0.4
    if which == "ghat0":
        ghat = np.zeros_like(ghat)
    y, gin = oracle.linear_scan(x, ghat, W0, eta, gout=gout)
    np.testing.assert_allclose(y, np.einsum("umd,utd->utm", W0, x), rtol=0, atol=1e-13)
    np.testing.assert_allclose(gin, np.einsum("umd,utm->utd", W0, gout), rtol=0, atol=1e-13)


def test_linearity_in_ghat_and_eta():
    U, T, d, m = 2, 50, 16, 12
    x, g1, W0, gout = _rand_problem(31, U, T, d, m)
    g2 = _rng(32).standard_normal((U, T, m))
    base_y = np.einsum("umd,utd->utm", W0, x)
    base_g = np.einsum("umd,utm->utd", W0, gout)

    def corr(g, eta):
        y, gi = oracle.linear_scan(x, g, W0, eta, gout=gout)
        return y - base_y, gi - base_g

    a, b = 0.7, -1.3
    y12, g12 = corr(a * g1 + b * g2, 0.2)
    y1, gg1 = corr(g1, 0.2)
    y2, gg2 = corr(g2, 0.2)
    np.testing.assert_allclose(y12, a * y1 + b * y2, rtol=0, atol=1e-12)
    np.testing.assert_allclose(g12, a * gg1 + b * gg2, rtol=0, atol=1e-12)
    y3, g3 = corr(g1, 0.6)
    np.testing.assert_allclose(y3, 3.0 * y1, rtol=0, atol=1e-12)
    np.testing.assert_allclose(g3, 3.0 * gg1, rtol=0, atol=1e-12)


def test_units_are_independent():
    """Each unit uses only its own W0 and its own history."""
    x, ghat, W0, gout = _rand_problem(41, 3, 20, 8, 8)
    y, gin = oracle.linear_scan(x, ghat, W0, 0.3, gout=gout)
    for u in range(3):
        yu, gu = oracle.linear_scan(x[u:u + 1], ghat[u:u + 1], W0[u:u + 1], 0.3,
                                    gout=gout[u:u + 1])
        np.testing.assert_array_equal(yu[0], y[u])
        np.testing.assert_array_equal(gu[0], gin[u])


# --------------------------------------------------------------- Theorem 1
def test_theorem1_recovery_linear():
    """A true serial learner with l_t = 1/2 ||y_t - c_t||^2 (so g_t = y_t - c_t),
    written independently here, is reproduced when its costates are supplied."""
    T, d, m = 64, 10, 6
    r = _rng(77)
    x = r.standard_normal((T, d))
    c = r.standard_normal((T, m))
    W0 = r.standard_normal((m, d)) * 0.3
    eta = 0.05
    W = W0.copy()
    ys, gs, gxs = [], [], []
    for t in range(T):
        yt = W @ x[t]
        gt = yt - c[t]
        ys.append(yt)
        gs.append(gt)
        gxs.append(W.T @ gt)       # dl_t/dx_t at the pre-update weights
        W = W - eta * np.outer(gt, x[t])
    g = np.array(gs)
    y, gin = oracle.linear_scan(x[None], g[None], W0, eta, gout=g[None])
    assert np.abs(y[0] - np.array(ys)).max() < 1e-13
    assert np.abs(gin[0] - np.array(gxs)).max() < 1e-13
    # Consistency residual ghat - g_tilde is zero at the fixed point (Theorem 1).
    assert np.abs(y[0] - c - g).max() < 1e-13


def _read_golden(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.split()
                vals[k] = float(v)
    return vals


def _sigmoid(v):
    return 1.0 / (1.0 + np.exp(-v))


def _e1_serial(seed):
    """Sec. 4.1 / Appendix B protocol: serial TTT of y = W2 tanh(W1 x), l = 1/2||y-c||^2,
    both matrices updated after every token with centered decay.  Manual backprop."""
    r = np.random.default_rng(seed)
    T, d, m, k = 32, 4, 7, 3
    W10 = r.standard_normal((m, d)) * (0.5 / np.sqrt(4))
    W20 = r.standard_normal((k, m)) * (0.5 / np.sqrt(7))
    va = r.standard_normal(d) * 0.25
    vm = r.standard_normal(d) * 0.25
    x = r.standard_normal((T, d))
    c = r.standard_normal((T, k))
    alpha = _sigmoid(x @ va + 1.5)
    mu = _sigmoid(x @ vm - 0.2)
    eta1, eta2 = mu / 4.0, mu / 7.0
    W1, W2 = W10.copy(), W20.copy()
    rec = {k_: [] for k_ in ("y", "gy", "gz", "gW1", "gz_ctrl", "gW1_ctrl")}
    for t in range(T):
        z = W1 @ x[t]
        h = np.tanh(z)
        y = W2 @ h
        gy = y - c[t]
        gz = (1.0 - h * h) * (W2.T @ gy)
        gz_ctrl = (1.0 - h * h) * (W20.T @ gy)     # "slow transpose only" control
        rec["y"].append(y)
        rec["gy"].append(gy)
        rec["gz"].append(gz)
        rec["gW1"].append(np.outer(gz, x[t]))
        rec["gz_ctrl"].append(gz_ctrl)
        rec["gW1_ctrl"].append(np.outer(gz_ctrl, x[t]))
        W1n = W10 + alpha[t] * (W1 - W10) - eta1[t] * np.outer(gz, x[t])
        W2n = W20 + alpha[t] * (W2 - W20) - eta2[t] * np.outer(gy, h)
        W1, W2 = W1n, W2n
    rec = {k_: np.array(v) for k_, v in rec.items()}
    return dict(x=x, W10=W10, W20=W20, alpha=alpha, eta1=eta1, eta2=eta2, **rec)


def _e1_parallel(p):
    """Appendix C explicit causal sums (the parallel construction) for the same MLP,
    fed the serial learner's costates (Appendix A eqs. scan1-reconstructed-reverse)."""
    x, alpha = p["x"], p["alpha"]
    T = x.shape[0]
    la = np.concatenate([[0.0], np.cumsum(np.log(alpha))])
    disc = np.zeros((T, T))
    for t in range(T):
        for i in range(t):
            disc[t, i] = np.exp(la[t] - la[i + 1])
    G1 = disc * p["eta1"][None, :]
    G2 = disc * p["eta2"][None, :]
    z = x @ p["W10"].T - (G1 * (x @ x.T)) @ p["gz"]
    h = np.tanh(z)
    y = h @ p["W20"].T - (G2 * (h @ h.T)) @ p["gy"]
    gh = p["gy"] @ p["W20"] - (G2 * (p["gy"] @ p["gy"].T)) @ h
    gz = (1.0 - h * h) * gh
    return y, gz


@pytest.mark.parametrize("seed", [17, 42, 123])
def test_e1_mlp_recovery_sec41(seed):
    gold = _read_golden("e1_recovery.txt")
    p = _e1_serial(seed)
    # (a) the dense causal-sum construction recovers serial TTT at rounding level
    y_par, gz_par = _e1_parallel(p)
    err_y = np.abs(y_par - p["y"]).max()
    err_gz = np.abs(gz_par - p["gz"]).max()
    err_gw = np.abs(gz_par[:, :, None] * p["x"][:, None, :] - p["gW1"]).max()
    assert max(err_y, err_gz, err_gw) < gold["rounding_bound"]
    # (b) the oracle, fed the same costates, recovers it too
    o = oracle.mlp_scan(p["x"][None], p["gz"][None], p["gy"][None], p["W10"], p["W20"],
                        p["eta1"], p["eta2"], act=oracle.ACT_TANH, alpha=p["alpha"],
                        gout=p["gy"][None])
    assert np.abs(o["y"][0] - p["y"]).max() < gold["rounding_bound"]
    assert np.abs(o["gz"][0] - p["gz"]).max() < gold["rounding_bound"]
    gw = o["gz"][0][:, :, None] * p["x"][:, None, :]
    assert np.abs(gw - p["gW1"]).max() < gold["rounding_bound"]
    # (c) the slow-transpose control changes the reverse by O(0.1-1)
    ctrl_gz = np.abs(p["gz_ctrl"] - p["gz"]).max()
    ctrl_gw = np.abs(p["gW1_ctrl"] - p["gW1"]).max()
    assert gold["control_min"] < max(ctrl_gz, ctrl_gw) < gold["control_max"]


def test_e1_control_over_three_seeds():
    """Maxima over the three seeds, as Fig. 2 reports them."""
    gold = _read_golden("e1_recovery.txt")
    cg, cw = 0.0, 0.0
    for seed in (17, 42, 123):
        p = _e1_serial(seed)
        cg = max(cg, np.abs(p["gz_ctrl"] - p["gz"]).max())
        cw = max(cw, np.abs(p["gW1_ctrl"] - p["gW1"]).max())
    assert gold["control_min"] < cg < gold["control_max"]
    assert gold["control_min"] < cw < gold["control_max"]


# ------------------------------------------------------------ MLP chaining
@pytest.mark.parametrize("act", [oracle.ACT_GELU_TANH, oracle.ACT_GELU_ERF, oracle.ACT_TANH])
def test_mlp_equals_two_chained_linear_maps(act):
    """Appendix A: layer 1 then sigma then layer 2 forward; costate through layer 2,
    sigma', then layer 1.  Composing the single-map oracle reproduces the MLP oracle."""
    U, T, d, m = 2, 40, 6, 10
    r = _rng(90 + act)
    x = r.standard_normal((U, T, d))
    ghz = r.standard_normal((U, T, m)) * 0.2
    ghy = r.standard_normal((U, T, d)) * 0.2
    W10 = r.standard_normal((m, d)) / np.sqrt(d)
    W20 = r.standard_normal((d, m)) / np.sqrt(m)
    gout = r.standard_normal((U, T, d))
    o = oracle.mlp_scan(x, ghz, ghy, W10, W20, 0.1, 0.05, act=act, gout=gout)
    z, _ = oracle.linear_scan(x, ghz, W10, 0.1)
    h = oracle.act(act, z)
    y, gh = oracle.linear_scan(h, ghy, W20, 0.05, gout=gout)
    gz = oracle.act_deriv(act, z) * gh
    _, gx = oracle.linear_scan(x, ghz, W10, 0.1, gout=gz)
    for a, b in ((o["z"], z), (o["h"], h), (o["y"], y), (o["gh"], gh), (o["gz"], gz),
                 (o["gx"], gx)):
        np.testing.assert_allclose(a, b, rtol=0, atol=1e-12)


# ------------------------------------------------------------- activations
@pytest.mark.parametrize("act", [oracle.ACT_GELU_TANH, oracle.ACT_GELU_ERF, oracle.ACT_TANH])
def test_activation_derivative_matches_finite_differences(act):
    z = np.linspace(-6, 6, 241)
    h = 1e-5
    fd = (oracle.act(act, z + h) - oracle.act(act, z - h)) / (2 * h)
    np.testing.assert_allclose(oracle.act_deriv(act, z), fd, rtol=0, atol=1e-8)


def test_activation_values():
    from scipy.special import erf
    z = np.linspace(-5, 5, 101)
    # GELU with the exact Gaussian CDF: z * Phi(z) (library erf).
    np.testing.assert_allclose(oracle.act(oracle.ACT_GELU_ERF, z),
                               z * 0.5 * (1 + erf(z / np.sqrt(2))), rtol=0, atol=1e-14)
    np.testing.assert_allclose(oracle.act(oracle.ACT_TANH, z), np.tanh(z), rtol=0, atol=1e-15)
    # The tanh approximation stays within 1e-3 of the exact GELU (a known bound).
    assert np.abs(oracle.act(oracle.ACT_GELU_TANH, z) - oracle.act(oracle.ACT_GELU_ERF, z)).max() < 1e-3
    assert oracle.act(oracle.ACT_GELU_TANH, np.array([0.0]))[0] == 0.0
    assert abs(oracle.act_deriv(oracle.ACT_GELU_TANH, np.array([0.0]))[0] - 0.5) < 1e-15
    np.testing.assert_allclose(oracle.act(oracle.ACT_NONE, z), z)
    np.testing.assert_allclose(oracle.act_deriv(oracle.ACT_NONE, z), np.ones_like(z))


# -------------------------------------------------------------- deployment
@pytest.mark.parametrize("seed", [17, 42])
def test_mlp_deploy_matches_serial_learner(seed):
    """Deployment (Sec. 3; Appendix A) writes actual costates, not proposals: layer 2
    writes the supplied gout_t and layer 1 its own reconstructed gz_t.  The hand-written serial
    learner of Sec. 4.1 does exactly that, so the deployed oracle reproduces it."""
    p = _e1_serial(seed)
    o = oracle.mlp_deploy(p["x"][None], p["W10"], p["W20"], p["eta1"], p["eta2"],
                          gout=p["gy"][None], act=oracle.ACT_TANH, alpha=p["alpha"])
    assert np.abs(o["y"][0] - p["y"]).max() < 1e-13
    assert np.abs(o["gz"][0] - p["gz"]).max() < 1e-13


def test_mlp_deploy_is_the_fixed_point_of_proposals():
    """Theorem 1: the reconstructed costate at token t depends only on proposals
    before t, so sweeping G <- F(G) from zero proposals fixes one more token per
    sweep and reaches the deployed learner's costates after T sweeps."""
    U, T, d, m, k = 2, 12, 5, 9, 4
    r = _rng(321)
    x = r.standard_normal((U, T, d))
    gout = r.standard_normal((U, T, k)) * 0.5
    W10 = r.standard_normal((m, d)) / np.sqrt(d)
    W20 = r.standard_normal((k, m)) / np.sqrt(m)
    eta1, eta2 = 0.2, 0.1
    dep = oracle.mlp_deploy(x, W10, W20, eta1, eta2, gout=gout, act=oracle.ACT_GELU_TANH)
    ghz = np.zeros((U, T, m))
    for n in range(1, T + 1):
        o = oracle.mlp_scan(x, ghz, gout, W10, W20, eta1, eta2, act=oracle.ACT_GELU_TANH,
                            gout=gout)
        ghz = o["gz"]
        assert np.abs(ghz[:, :n] - dep["gz"][:, :n]).max() < 1e-12
        if n <= 3:  # later tokens still see a wrong history (the gap shrinks every sweep)
            assert np.abs(ghz[:, n:] - dep["gz"][:, n:]).max() > 1e-9
    for key in ("z", "h", "y", "gh", "gx"):
        assert np.abs(o[key] - dep[key]).max() < 1e-12, key


# ------------------------------------------------- consistency term (Eq. 5)
def test_consistency_hand_values():
    """||ghat - gtilde||^2 / w on vectors small enough to add by hand."""
    p = np.array([[[1.0, 2.0, 3.0, 4.0], [0.5, -0.5, 0.0, 2.0]]])
    g = np.array([[[0.0, 2.0, 5.0, 4.0], [0.5, 0.5, 0.0, -1.0]]])
    c = oracle.consistency(p, g)
    assert c.shape == (1, 2)
    assert c[0, 0] == (1.0 + 0.0 + 4.0 + 0.0) / 4.0
    assert c[0, 1] == (0.0 + 1.0 + 0.0 + 9.0) / 4.0
    assert np.all(oracle.consistency(g, g) == 0.0)


def test_consistency_vanishes_at_the_serial_learner():
    """Theorem 1: with the deployed learner's own costates as proposals, the costates
    the scans reconstruct equal the proposals, so both terms of the MLP consistency
    loss (Appendix A) vanish; a proposal perturbed at one token raises the layer-1
    term there by exactly ||perturbation||^2 / m and leaves every earlier token at 0."""
    U, T, d, m, k = 2, 10, 5, 7, 3
    r = _rng(77)
    x = r.standard_normal((U, T, d))
    gout = r.standard_normal((U, T, k)) * 0.5
    W10 = r.standard_normal((m, d)) / np.sqrt(d)
    W20 = r.standard_normal((k, m)) / np.sqrt(m)
    eta1, eta2 = 0.3, 0.2
    dep = oracle.mlp_deploy(x, W10, W20, eta1, eta2, gout=gout, act=oracle.ACT_GELU_TANH)
    o = oracle.mlp_scan(x, dep["gz"], gout, W10, W20, eta1, eta2, act=oracle.ACT_GELU_TANH,
                        gout=gout)
    assert oracle.consistency(dep["gz"], o["gz"]).max() < 1e-28
    assert oracle.consistency(gout, gout).max() == 0.0
    t0 = 4
    bump = np.zeros((U, T, m))
    bump[:, t0] = r.standard_normal((U, m))
    o2 = oracle.mlp_scan(x, dep["gz"] + bump, gout, W10, W20, eta1, eta2,
                         act=oracle.ACT_GELU_TANH, gout=gout)
    c2 = oracle.consistency(dep["gz"] + bump, o2["gz"])
    assert c2[:, :t0].max() < 1e-28
    # token t0's reconstruction reads only writes before t0, so it is unchanged
    expect = (bump[:, t0] ** 2).sum(axis=-1) / m
    assert np.allclose(c2[:, t0], expect, rtol=1e-12, atol=0)


# ------------------------------------------------------ suffix read (gradients)
def test_suffix_scan_brute_force():
    """r_s = sum_{t>s} (k_t . q_s) v_t written as the double sum; r_{T-1} = 0."""
    U, T, dq, dv = 2, 9, 3, 4
    r = _rng(401)
    q, k, v = r.standard_normal((U, T, dq)), r.standard_normal((U, T, dq)), r.standard_normal((U, T, dv))
    out = oracle.suffix_scan(q, k, v)
    ref = np.zeros((U, T, dv))
    for u in range(U):
        for s in range(T):
            for t in range(s + 1, T):
                ref[u, s] += np.dot(k[u, t], q[u, s]) * v[u, t]
    assert np.abs(out - ref).max() < 1e-13
    assert np.abs(out[:, -1]).max() == 0.0


def _fd_eta(loss, eta, h=1e-3):
    g = np.empty_like(eta)
    for s in range(eta.shape[0]):
        e1, e2 = eta.copy(), eta.copy()
        e1[s] += h
        e2[s] -= h
        g[s] = (loss(e1) - loss(e2)) / (2 * h)
    return g


def test_eta_gradient_of_forward_read_is_a_suffix_read():
    """y_t is linear in every eta_s (unit retention), so central differences of
    the sequential learner give dL/deta_s exactly (up to rounding); with
    L = sum_t u_t . y_t they equal -ghat_s . r_s, r the suffix read with q = k = x, v = u."""
    T, d, m = 24, 5, 7
    r = _rng(402)
    x, gh, u = r.standard_normal((1, T, d)), r.standard_normal((1, T, m)), r.standard_normal((1, T, m))
    W0 = r.standard_normal((m, d)) * 0.3
    eta = r.uniform(0.01, 0.2, T)
    loss = lambda e: float(np.sum(u * oracle.linear_scan(x, gh, W0, e)[0]))
    fd = _fd_eta(loss, eta)
    rs = oracle.suffix_scan(x, x, u)[0]
    an = -np.sum(gh[0] * rs, axis=1)
    assert np.abs(fd - an).max() < 1e-7 * max(1.0, np.abs(an).max())


def test_eta_gradient_of_costate_read_is_a_suffix_read():
    """gin_t = W_t^T g_t: with L = sum_t w_t . gin_t, dL/deta_s = -x_s . r_s where r is
    the suffix read with q = ghat, k = g_out, v = w."""
    T, d, m = 20, 6, 4
    r = _rng(403)
    x, gh, go = r.standard_normal((1, T, d)), r.standard_normal((1, T, m)), r.standard_normal((1, T, m))
    w = r.standard_normal((1, T, d))
    W0 = r.standard_normal((m, d)) * 0.3
    eta = r.uniform(0.01, 0.2, T)
    loss = lambda e: float(np.sum(w * oracle.linear_scan(x, gh, W0, e, gout=go, want_y=False)[1]))
    fd = _fd_eta(loss, eta)
    rs = oracle.suffix_scan(gh, go, w)[0]
    an = -np.sum(x[0] * rs, axis=1)
    assert np.abs(fd - an).max() < 1e-7 * max(1.0, np.abs(an).max())


# ------------------------------------------------------ gate derivatives
def _gate_case(seed, T, d, m):
    r = _rng(seed)
    x, gh = r.standard_normal((1, T, d)), r.standard_normal((1, T, m))
    go, u, w = r.standard_normal((1, T, m)), r.standard_normal((1, T, m)), r.standard_normal((1, T, d))
    W0 = r.standard_normal((m, d)) * 0.3
    eta = r.uniform(0.01, 0.3, T)
    alpha = r.uniform(0.5, 1.0, T)
    alpha[T // 3] = 0.0     # a reset
    alpha[T // 2] = -0.6    # a negative retention
    return x, gh, go, u, w, W0, eta, alpha


def _fd(loss, v, h=1e-4):
    g = np.empty_like(v)
    for s in range(v.shape[0]):
        v1, v2 = v.copy(), v.copy()
        v1[s] += h
        v2[s] -= h
        g[s] = (loss(v1) - loss(v2)) / (2 * h)
    return g


@pytest.mark.parametrize("read", ["forward", "costate"])
def test_gate_grads_match_central_differences(read):
    """Every read is affine in each single alpha_j and eta_j (each decay product holds
    alpha_j at most once), so central differences of the sequential learner give
    dL/dalpha_j and dL/deta_j up to rounding.  Non-square maps catch a transposed
    operand; a reset and a negative retention are included."""
    T, d, m = 26, 5, 3
    x, gh, go, u, w, W0, eta, alpha = _gate_case(404 if read == "forward" else 405, T, d, m)
    if read == "forward":
        loss = lambda e, a: float(np.sum(u * oracle.linear_scan(x, gh, W0, e, alpha=a)[0]))
        ga, ge = oracle.gate_grads(x, gh, eta, alpha, u, x)
    else:
        loss = lambda e, a: float(np.sum(
            w * oracle.linear_scan(x, gh, W0, e, alpha=a, gout=go, want_y=False)[1]))
        ga, ge = oracle.gate_grads(x, gh, eta, alpha, go, w)
    fd_a = _fd(lambda a: loss(eta, a), alpha) * alpha
    fd_e = _fd(lambda e: loss(e, alpha), eta)
    scale = max(1.0, np.abs(fd_a).max(), np.abs(fd_e).max())
    assert np.abs(ga[0] - fd_a).max() < 1e-8 * scale
    assert np.abs(ge[0] - fd_e).max() < 1e-8 * scale


def test_gate_grads_brute_force_pairs():
    """alpha_j dL/dalpha_j is the sum, over every write i and later read s with
    i < j < s, of that pair's contribution -eta_i prod_{i<r<s} alpha_r
    (u_s . ghat_i)(x_i . x_s) to L = sum_s u_s . y_s; dL/deta_i is the sum of the
    same contributions over s > i, divided by eta_i."""
    T, d, m = 7, 3, 2
    x, gh, go, u, w, W0, eta, alpha = _gate_case(406, T, d, m)
    ga, ge = oracle.gate_grads(x, gh, eta, alpha, u, x)
    c = np.zeros((T, T))
    for i in range(T):
        for s_ in range(i + 1, T):
            c[i, s_] = -eta[i] * np.prod(alpha[i + 1:s_]) * np.dot(u[0, s_], gh[0, i]) * np.dot(x[0, i], x[0, s_])
    ref_a = np.array([sum(c[i, s_] for i in range(j) for s_ in range(j + 1, T)) for j in range(T)])
    ref_e = np.array([c[i, i + 1:].sum() / eta[i] for i in range(T)])
    assert np.abs(ga[0] - ref_a).max() < 1e-12 * max(1.0, np.abs(ref_a).max())
    assert np.abs(ge[0] - ref_e).max() < 1e-12 * max(1.0, np.abs(ref_e).max())
    assert ga[0, 0] == 0.0 and ga[0, -1] == 0.0 and ge[0, -1] == 0.0


def test_gate_grads_at_unit_retention_are_the_suffix_read():
    """With alpha = 1 the decayed suffix read is the plain suffix read: dL/deta_j =
    -ghat_j . r_j with r = suffix_scan(x, x, u) (a separate routine)."""
    T, d, m = 30, 4, 6
    x, gh, go, u, w, W0, eta, alpha = _gate_case(407, T, d, m)
    ga, ge = oracle.gate_grads(x, gh, eta, np.ones(T), u, x)
    rs = oracle.suffix_scan(x, x, u)[0]
    an = -np.sum(gh[0] * rs, axis=1)
    assert np.abs(ge[0] - an).max() < 1e-12 * max(1.0, np.abs(an).max())


def test_gate_grads_telescoping_identity():
    """alpha_j dL/dalpha_j = sum_{t>j} (A_t - B_t) - B_j with A_t = u_t . (y_t - W0 x_t)
    (the pairs ending at read t) and B_t = eta_t dL/deta_t (the pairs starting at
    write t): the pairs that straddle j, counted another way."""
    T, d, m = 40, 5, 4
    x, gh, go, u, w, W0, eta, alpha = _gate_case(408, T, d, m)
    ga, ge = oracle.gate_grads(x, gh, eta, alpha, u, x)
    y = oracle.linear_scan(x, gh, W0, eta, alpha=alpha)[0][0]
    A = np.sum(u[0] * (y - x[0] @ W0.T), axis=1)
    B = eta * ge[0]
    D = A - B
    ref = np.array([D[j + 1:].sum() - B[j] for j in range(T)])
    assert np.abs(ga[0] - ref).max() < 1e-11 * max(1.0, np.abs(ref).max())


def test_gated_learner_property_sweep():
    """Random shapes and gates (zeros, negative retention, document cuts) against the
    closed form of Eq. 2, restricted to each document."""
    hyp = pytest.importorskip("hypothesis")
    st = pytest.importorskip("hypothesis.strategies")

    @hyp.settings(max_examples=60, deadline=None, derandomize=True)
    @hyp.given(T=st.integers(1, 12), d=st.integers(1, 5), m=st.integers(1, 5),
               seed=st.integers(0, 10_000), n_cuts=st.integers(0, 3))
    def check(T, d, m, seed, n_cuts):
        r = _rng(seed)
        x, ghat, W0, gout = _rand_problem(seed, 1, T, d, m)
        eta = r.uniform(0.0, 0.6, T)
        alpha = r.uniform(-1.0, 1.0, T)
        alpha[r.random(T) < 0.25] = 0.0
        cuts = sorted(set(int(c) for c in r.integers(1, max(T, 2), n_cuts) if 0 < c < T))
        y, gin = oracle.linear_scan_docs(x, ghat, W0, eta, _doc_starts(T, cuts), alpha=alpha,
                                         gout=gout)
        bounds = [0, *cuts, T]
        for a, b in zip(bounds[:-1], bounds[1:]):
            for t in range(a, b):
                W_t = W0[0] + _closed_form_delta(t - a, x[0, a:b], ghat[0, a:b], eta[a:b],
                                                 alpha[a:b])
                np.testing.assert_allclose(y[0, t], W_t @ x[0, t], rtol=0, atol=1e-13)
                np.testing.assert_allclose(gin[0, t], W_t.T @ gout[0, t], rtol=0, atol=1e-13)

    check()
