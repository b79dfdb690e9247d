"""The rescaled accumulation that the capture kernels use is an exact rearrangement of
Eq. 1's recurrence: written out here in fp64 (with the kernels' renormalisation rules:
an exponent window, a token count, tokens applied directly when their own step leaves the
window), it reproduces the oracle's token-by-token rollout to rounding. CPU only; this
checks the algebra the kernels rely on, not the kernels."""
import numpy as np
import pytest

import oracle
import synth

LOG2E = 1.0 / np.log(2.0)


def _real_rescaled(x, dt, a0, B, lmax=6.0, group=4):
    """A[d, n] = (n+1) a0[d]: h_n = E^-(n+1) G_n, E = 2^L, L = sum dt (-a0 log2 e).

    The D channels decide together, as the lanes of one warp do: tokens go in groups;
    when some channel's exponent would leave the window at the group's end, every channel
    moves to the bottom of the window (L = -lmax) before the group. A negative dt in the
    group, or a group whose own increment exceeds the window, goes token by token: there
    a channel leaving [-lmax, lmax] makes all restart from L = 0, and a token whose own
    step leaves the window is applied directly."""
    T, D = x.shape
    N = B.shape[1]
    n1 = np.arange(1, N + 1)
    k = -a0 * LOG2E
    G, L = np.zeros((D, N)), np.zeros(D)

    def token_checked(t):
        nonlocal G, L
        u = dt[t] * x[t]
        Ln = L + dt[t] * k
        if (np.abs(Ln) > lmax).any():
            G, L = G * 2.0 ** (-L[:, None] * n1), np.zeros(D)    # renormalise: G = h
            Ln = dt[t] * k
            own = np.abs(Ln) > lmax                               # the token's own step: direct
            G[own] = G[own] * 2.0 ** (-Ln[own, None] * n1) + u[own, None] * B[t]
            u = np.where(own, 0.0, u)
            Ln = np.where(own, 0.0, Ln)
        G = G + u[:, None] * 2.0 ** (Ln[:, None] * n1) * B[t]
        L = Ln

    t = 0
    while t + group <= T:
        Lk = L + np.cumsum(dt[t:t + group] * k, axis=0)
        slow = False
        if (Lk[-1] > lmax).any() or (dt[t:t + group] < 0).any():
            slow = bool((dt[t:t + group] < 0).any())
            if not slow:
                G = G * 2.0 ** (-(L + lmax)[:, None] * n1)           # frame to the window's bottom
                L = np.full(D, -lmax)
                Lk = L + np.cumsum(dt[t:t + group] * k, axis=0)
                slow = bool((Lk[-1] > lmax).any())
        if slow:
            for tt in range(t, t + group):
                token_checked(tt)
        else:
            for j in range(group):
                u = dt[t + j] * x[t + j]
                G = G + u[:, None] * 2.0 ** (Lk[j][:, None] * n1) * B[t + j]
            L = Lk[-1]
        t += group
    for tt in range(t, T):
        token_checked(tt)
    return G * 2.0 ** (-L[:, None] * n1)


def _complex_rescaled(x, dt, A_re, A_im, B, power):
    """Power form (A_re[n] = (n+1) A_re[0]) or harmonic form (any A_re): P_n = M_n Z^n,
    h_n = P_n G_n; renormalised on the exponent window and every 64 tokens."""
    T, D = x.shape
    N = B.shape[1]
    n = np.arange(N)
    out = np.zeros((D, N), complex)
    for d in range(D):
        c = A_re[d] * LOG2E                               # log2 of the per-unit-dt decay, per index
        a1 = A_im[d, 1]
        G, S, phi, since = np.zeros(N, complex), 0.0, 0.0, 0

        def P(S, phi):                                    # decay product since the last renormalisation
            return 2.0 ** (S * c) * np.exp(1j * phi * n)
        for t in range(T):
            u = dt[t, d] * x[t, d]
            Sn, ph = S + dt[t, d], phi + dt[t, d] * a1
            wide = np.max(np.abs(Sn * c)) > 96.0 if not power else abs(Sn * c[0]) > 6.0
            if wide or since >= 64:
                G, S, phi, since = P(S, phi) * G, 0.0, 0.0, 0
                Sn, ph = dt[t, d], dt[t, d] * a1
                own = np.max(np.abs(Sn * c)) > 96.0 if not power else abs(Sn * c[0]) > 6.0
                if own:
                    G = P(Sn, ph) * G + u * B[t]
                    since += 1
                    continue
            G = G + u * B[t] / P(Sn, ph)
            S, phi, since = Sn, ph, since + 1
        out[d] = P(S, phi) * G
    return out


@pytest.mark.parametrize("scale", [1.0, 0.01, 30.0, -1.0])
def test_real_rescaled_equals_rollout(scale):
    T, D, N = 301, 4, 16
    x, dt, _, B, _ = synth.host_scan_inputs(T, D, N, seed=41)
    dt = dt.astype(np.float64) * abs(scale)
    if scale < 0:
        # a few negative steps: those groups go token by token
        dt[np.random.default_rng(42).random(dt.shape) < 0.02] *= -1.0
    a0 = -np.array([1.0, 0.3, 2.0, 0.05])
    A = a0[:, None] * np.arange(1, N + 1)[None, :]
    ref, _ = oracle.scan(x, dt, A, B, [0, T])
    got = _real_rescaled(x.astype(np.float64), dt, a0, B.astype(np.float64))
    np.testing.assert_allclose(got, ref[0], rtol=1e-9, atol=1e-12 * np.abs(ref).max())


@pytest.mark.parametrize("power", [True, False])
@pytest.mark.parametrize("scale", [1.0, 0.01, 30.0])
def test_complex_rescaled_equals_rollout(power, scale):
    T, D, N = 300, 3, 16
    x, dt, _, B, _ = synth.host_scan_inputs(T, D, N, seed=43)
    dt = dt.astype(np.float64) * scale
    rng = np.random.default_rng(44)
    if power:
        A_re = -synth.softplus_np(rng.standard_normal(D))[:, None] * np.arange(1, N + 1)[None, :]
    else:
        A_re = -synth.softplus_np(rng.standard_normal((D, N)))
    A_im = np.pi * (1.0 + 0.1 * rng.standard_normal(D))[:, None] * np.arange(N)[None, :]
    ref, _ = oracle.scan_complex(x, dt, A_re, A_im, B, [0, T])
    got = _complex_rescaled(x.astype(np.float64), dt, A_re, A_im, B.astype(np.float64), power)
    np.testing.assert_allclose(got, ref[0], rtol=1e-9, atol=1e-12 * np.abs(ref).max())
