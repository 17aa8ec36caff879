"""Cutoff-distribution design (oracle, float64): score proxy, timestep weights, budgeted
monotone xi, and the integer masses the sampler takes.

Section 3.3 and Appendix D: the output-head score proxy of a token is
    gamma_t = ||h_t||^2 (1 - 2 p_t(o_t) + ||p_t||^2),
the squared Frobenius norm of d log p(o_t) / dW = (e_o - p) h^T.
Section 3.3 (Eq. wtilde_factorized1): per prompt, gamma_bar_t averages gamma_t over the
group's rollouts at step t; the timestep weight is w_t = gamma_bar_t * u_t, with u_t the
reward-uncertainty proxy (an input here).
Appendix F: minimise sum_t w_t / xi_t subject to sum_t xi_t = B and 1 >= xi_1 >= ... >= xi_T.
Without monotonicity, xi_t = B sqrt(w_t) / sum_j sqrt(w_j). With it, the optimum is constant on
contiguous blocks with scores s_m = sqrt(W_m / L_m) and xi_m = B s_m / sum_j L_j s_j; pooling
adjacent violators (PAV) until the scores are non-increasing gives the monotone optimum. With the
cap xi <= 1, a prefix of coordinates saturates at 1 and the same solution applies to the rest
with the budget reduced by the prefix length.
Section 4 (Baselines): the cutoff variants Uniform, Time prior xi_t = exp(-lambda (t-1)),
Heuristic (closed form, then the running minimum), and the fixed prefix of length L.

Masses: Pr(H = h) = xi_h - xi_{h+1} (xi_{T+1} = 0) and Pr(H = 0) = 1 - xi_1, quantised to
integers q_h = floor(Pr(H = h) 2^62); the deficit 2^62 - sum_h q_h is the mass of H = 0.
"""
from __future__ import annotations

import math

import numpy as np

ONE62 = 1 << 62


# ----------------------------------------------------------------------------- score proxy
def score_proxy(H, W, tok):
    """gamma_t = ||h_t||^2 ||e_o - p_t||^2 and log p_t(o_t) for every row (Appendix D; the paper's
    1 - 2 p(o) + ||p||^2 is ||e_o - p||^2 expanded)."""
    H = np.asarray(H, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    tok = np.asarray(tok)
    gamma = np.empty(len(tok))
    logp = np.empty(len(tok))
    for r0 in range(0, len(tok), 128):
        z = H[r0:r0 + 128] @ W.T
        m = z.max(axis=1, keepdims=True)
        e = np.exp(z - m)
        p = e / e.sum(axis=1, keepdims=True)
        rows = np.arange(z.shape[0])
        po = p[rows, tok[r0:r0 + 128]]
        hn = (H[r0:r0 + 128] ** 2).sum(axis=1)
        resid = -p                                   # e_o - p, written out: no cancellation near p(o) = 1
        resid[rows, tok[r0:r0 + 128]] += 1.0
        gamma[r0:r0 + 128] = hn * (resid * resid).sum(axis=1)
        logp[r0:r0 + 128] = np.log(po)
    return gamma, logp


# ----------------------------------------------------------------------------- weights
def group_mean_by_step(values_full, L, K):
    """gamma_bar[p][t-1] = (1/K) sum over the group's completions that reach step t.

    Completions shorter than t contribute 0 (their score at t is zero): the average is over all
    K rollouts. values_full is laid out completion after completion (unpacked batch order).
    Sums run sequentially over k in float64.
    """
    L = np.asarray(L)
    B = len(L)
    P = B // K
    T_max = int(L.max())
    off = np.concatenate([[0], np.cumsum(L)])
    out = np.zeros((P, T_max))
    for p in range(P):
        acc = [0.0] * T_max
        for j in range(K):
            k = p * K + j
            seg = values_full[off[k]:off[k] + L[k]]
            for t in range(int(L[k])):
                acc[t] = acc[t] + float(seg[t])
        out[p] = [a / K for a in acc]
    return out


# ----------------------------------------------------------------------------- design
def closed_form(w, B):
    """Unconstrained optimum xi_t = B sqrt(w_t) / sum_j sqrt(w_j) (Appendix F)."""
    r = [math.sqrt(float(x)) for x in w]
    tot = 0.0
    for x in r:
        tot += x
    return np.array([B * x / tot for x in r])


def pav_blocks(w):
    """Pool adjacent violators: blocks (start, length, W) whose scores sqrt(W / L) are non-increasing.

    Blocks are pushed left to right; while the last block's score is above the one before it
    (a violation of xi_1 >= xi_2 >= ...), the two are merged.
    """
    blocks = []  # [start, length, weight sum]
    for t, x in enumerate(w):
        blocks.append([t, 1, float(x)])
        while len(blocks) > 1 and math.sqrt(blocks[-2][2] / blocks[-2][1]) < math.sqrt(blocks[-1][2] / blocks[-1][1]):
            s, n, Wm = blocks.pop()
            blocks[-1][1] += n
            blocks[-1][2] += Wm
    return blocks


def monotone_design(w, B):
    """Monotone optimum without the cap: xi on PAV blocks, xi_m = B s_m / sum_j L_j s_j."""
    blocks = pav_blocks(w)
    s = [math.sqrt(Wm / n) for _, n, Wm in blocks]
    den = 0.0
    for (_, n, _), sm in zip(blocks, s):
        den += n * sm
    xi = np.empty(len(w))
    for (t0, n, _), sm in zip(blocks, s):
        xi[t0:t0 + n] = B * sm / den
    return xi


def capped_monotone_design(w, B):
    """Monotone optimum with xi <= 1: the smallest saturated prefix p for which the design of the
    suffix with budget B - p starts at or below 1 (Appendix F, remark on the cap)."""
    T = len(w)
    if not (0 < B <= T):
        raise ValueError("the budget must lie in (0, T]")
    for p in range(T):
        rest = monotone_design(w[p:], B - p)
        if rest[0] <= 1.0:
            return np.concatenate([np.ones(p), rest])
    return np.ones(T)


def heuristic_design(w, B):
    """Section 4 (Heuristic): closed form, then xi_t <- min(xi_{t-1}, xi_t); capped at 1."""
    xi = closed_form(w, B)
    for t in range(1, len(xi)):
        xi[t] = min(xi[t - 1], xi[t])
    return np.minimum(xi, 1.0)


def time_prior_design(T, B, iters=200):
    """Section 4 (Time prior): xi_t = exp(-lam (t-1)), with lam >= 0 chosen so sum_t xi_t = B."""
    if not (0 < B <= T):
        raise ValueError("the budget must lie in (0, T]")
    t = np.arange(T, dtype=np.float64)

    def budget(lam):
        return float(np.exp(-lam * t).sum())

    if budget(0.0) <= B:
        return np.ones(T)
    lo, hi = 0.0, 1.0
    while budget(hi) > B:
        hi *= 2.0
    for _ in range(iters):
        mid = 0.5 * (lo + hi)
        if budget(mid) > B:
            lo = mid
        else:
            hi = mid
    return np.exp(-hi * t)


def uniform_design(T):
    """Section 4 (Uniform): the cutoff is uniform on 1..T, so xi_t = (T - t + 1) / T."""
    return (T - np.arange(T, dtype=np.float64)) / T


def fixed_prefix_design(T, Lfix):
    """Section 4 (fixed prefix): H = min(Lfix, T) with probability 1 (biased control)."""
    return (np.arange(1, T + 1) <= Lfix).astype(np.float64)


def masses_from_xi(xi):
    """Integer masses q_h = floor((xi_h - xi_{h+1}) 2^62), h = 1..T; the deficit is Pr(H = 0).

    Rounding can make the differences add up to slightly more than xi_1; any excess over 2^62
    (only possible when xi_1 is 1) is taken from the largest mass, lowest index on ties.
    """
    T = len(xi)
    q = [0] * T
    for h in range(T):
        nxt = float(xi[h + 1]) if h + 1 < T else 0.0
        d = float(xi[h]) - nxt
        q[h] = int(math.floor(d * float(ONE62))) if d > 0.0 else 0
    excess = sum(q) - ONE62
    if excess > 0:
        i = max(range(T), key=lambda j: (q[j], -j))
        q[i] -= excess
    return np.array(q, dtype=np.uint64)


# ----------------------------------------------------------------------------- whole design step
STRATEGIES = ("optimized", "heuristic", "uniform", "time_prior", "fixed")
W_FLOOR = 1e-12   # weights below W_FLOOR * max_t w_t are raised to it, so every xi_t > 0


def timestep_weights(gamma_bar_p, u_p):
    """w_t = gamma_bar_t * u_t (u = 1 when not given), floored at W_FLOOR * max_t w_t so that the
    design keeps xi_t > 0 (Section 3.2 requires xi_T > 0); all-zero weights become all ones."""
    T = len(gamma_bar_p)
    w = [float(gamma_bar_p[t]) * (float(u_p[t]) if u_p is not None else 1.0) for t in range(T)]
    if not all(math.isfinite(x) for x in w):
        raise ValueError("non-finite timestep weight: the design is undefined")
    wmax = max(w)
    if not wmax > 0.0:
        return [1.0] * T
    fl = W_FLOOR * wmax
    return [x if x > fl else fl for x in w]


def design_cutoff_masses(L, K, gamma_full, u, B, strategy, param=0.0):
    """Masses q [P, T_max] (uint64) and xi [P, T_max] (float64) for every prompt.

    Prompt p's horizon is T_p = the longest completion of its group; its budget is min(B, T_p).
    optimized: capped monotone design of w; heuristic: closed form + running minimum + cap;
    uniform: xi_t = (T_p - t + 1) / T_p; time_prior: exp(-lam (t-1)) with sum_t xi_t = budget;
    fixed: xi_t = 1 for t <= param.
    """
    L = np.asarray(L)
    B_total = len(L)
    P = B_total // K
    T_max = int(L.max())
    gbar = group_mean_by_step(gamma_full, L, K) if strategy in ("optimized", "heuristic") else None
    q = np.zeros((P, T_max), dtype=np.uint64)
    xi_all = np.zeros((P, T_max))
    for p in range(P):
        Tp = int(L[p * K:(p + 1) * K].max())
        Bp = min(float(B), float(Tp))
        if strategy in ("optimized", "heuristic"):
            w = timestep_weights(gbar[p, :Tp], None if u is None else u[p, :Tp])
            xi = capped_monotone_design(w, Bp) if strategy == "optimized" else heuristic_design(w, Bp)
        elif strategy == "uniform":
            xi = uniform_design(Tp)
        elif strategy == "time_prior":
            xi = time_prior_design(Tp, Bp)
        elif strategy == "fixed":
            xi = fixed_prefix_design(Tp, int(param))
        else:
            raise ValueError(strategy)
        q[p, :Tp] = masses_from_xi(xi)
        xi_all[p, :Tp] = xi
    return q, xi_all


# ----------------------------------------------------------------------------- reward uncertainty
def topk_policy(H, W, k):
    """Per row, the k most likely next tokens of softmax(W h) and their probabilities (float64;
    ties go to the lower token id). Appendix I: the u_t estimate keeps the top k = 16."""
    H = np.asarray(H, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    idx = np.empty((H.shape[0], k), dtype=np.int64)
    prob = np.empty((H.shape[0], k))
    for r0 in range(0, H.shape[0], 128):
        z = H[r0:r0 + 128] @ W.T
        m = z.max(axis=1, keepdims=True)
        p = np.exp(z - m)
        p /= p.sum(axis=1, keepdims=True)
        order = np.lexsort((np.broadcast_to(np.arange(z.shape[1]), z.shape), -z), axis=1)[:, :k]
        idx[r0:r0 + 128] = order
        prob[r0:r0 + 128] = np.take_along_axis(p, order, axis=1)
    return idx, prob


def reward_uncertainty(L, K, R, top_idx, top_prob):
    """u[p][t-1] = 1/2 - 1/2 || p_hat pi_G(.|t) - (1 - p_hat) pi_B(.|t) ||_1 (Appendix E, Eq. ut_def),
    estimated from the group's K completions (Appendix E, last paragraph):

    p_hat = fraction of the group with R = 1 (R >= 0.5 counts as success); pi_G(.|t) / pi_B(.|t)
    average the old-policy next-token distributions at step t over the successful / unsuccessful
    completions that reach t (a class with none contributes 0). Each distribution is represented by
    its top-k tokens plus one "other" symbol holding its remaining mass (the top-k approximation of
    Appendix I; with k = V it is the definition). Rows of top_idx / top_prob are in completion order.
    Steps beyond the group's horizon get u = 0.
    """
    L = np.asarray(L)
    Bn = len(L)
    P = Bn // K
    T_max = int(L.max())
    off = np.concatenate([[0], np.cumsum(L)])
    u = np.zeros((P, T_max))
    for p in range(P):
        ks = list(range(p * K, (p + 1) * K))
        succ = [k for k in ks if float(R[k]) >= 0.5]
        fail = [k for k in ks if float(R[k]) < 0.5]
        p_hat = len(succ) / K
        Tp = int(max(L[k] for k in ks))
        for t in range(Tp):
            g_alive = [k for k in succ if L[k] > t]
            b_alive = [k for k in fail if L[k] > t]
            coef = {}
            for k in g_alive:
                coef[k] = p_hat / len(g_alive)
            for k in b_alive:
                coef[k] = -(1.0 - p_hat) / len(b_alive)
            mass = {}
            other = 0.0
            for k, c in coef.items():
                row = off[k] + t
                tot = 0.0
                for v, pv in zip(top_idx[row], top_prob[row]):
                    mass[int(v)] = mass.get(int(v), 0.0) + c * float(pv)
                    tot += float(pv)
                other += c * (1.0 - tot)
            l1 = sum(abs(x) for x in mass.values()) + abs(other)
            u[p, t] = min(0.5, max(0.0, 0.5 - 0.5 * l1))
    return u


# ---------------------------------------------------------------- continuous rewards (Appendix G)
LN2 = 0.6931471805599453          # the double nearest ln 2
SIGMOID_CLAMP = 40.0              # |r| beyond this decides no label differently (see below)


def sigmoid_recipe(r: float) -> float:
    """sigma(r) = 1 / (1 + e^(-r)) by one fixed sequence of IEEE double operations.

    With z = -r clamped to [-40, 40]: k = floor(z / ln2 + 1/2), f = z - k ln2 (|f| <= ln2 / 2 plus
    rounding), e^f by Horner's rule over its Taylor series to degree 16 (p <- 1 + f p / n for
    n = 16, ..., 1; the truncation error is below 1e-22), e^z = e^f 2^k, and sigma = 1 / (1 + e^z).
    Every step is a correctly rounded +, -, *, / or an exact power-of-two scaling, so the kernel
    that repeats the sequence gets the same double. The clamp moves sigma by less than 4.3e-18,
    below the 2^-53 resolution of the uniform it is compared with, so no label changes.
    """
    r = float(r)
    if r != r:
        return 0.0
    z = -r
    z = SIGMOID_CLAMP if z > SIGMOID_CLAMP else (-SIGMOID_CLAMP if z < -SIGMOID_CLAMP else z)
    k = math.floor(z / LN2 + 0.5)
    f = z - k * LN2
    p = 1.0
    for n in range(16, 0, -1):
        p = 1.0 + (f * p) / n
    e = math.ldexp(p, k)
    return 1.0 / (1.0 + e)


def binarize_rewards(R, seed: int, step: int, traj_base: int = 0) -> np.ndarray:
    """Appendix G: labels y_k ~ Bernoulli(sigma(R_k)) for the u_t estimate only (the update keeps
    the continuous R). Trajectory k draws u = m 2^-53 from the Philox stream keyed by
    (seed, "PSPPRWD1") at counter (traj_base + k, step, 0, 0), and y_k = 1 when u < sigma(R_k),
    i.e. when m < sigma 2^53 (a NaN reward gives 0). Returns float32 labels in {0, 1}.
    """
    from .philox import reward_uniform53
    R = np.asarray(R, dtype=np.float32)
    y = np.zeros(len(R), dtype=np.float32)
    for k, r in enumerate(R):
        m = reward_uniform53(seed, step, traj_base + k)
        y[k] = 1.0 if float(m) < sigmoid_recipe(float(r)) * 9007199254740992.0 else 0.0
    return y
