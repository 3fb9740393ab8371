"""Pins for the oracle's gradients in the saturated regime (probabilities near one-hot,
App. B): against 150-digit evaluations of the same softmax Jacobian (mpmath), for the
categorical relaxation and for a binary mask x sign instance.  A direct q_k - w~ loses
every digit here (w~ rounds to q_m), which is the failure these pins guard."""
import mpmath
import numpy as np

from oracle import gsq_oracle as O

mpmath.mp.dps = 150       # probabilities reach e^-120: 50 digits would cancel too


def _mp_softmax_grad(l, g, q, tau, kappa):
    z = [(kappa * mpmath.mpf(float(a)) + mpmath.mpf(float(b))) / tau for a, b in zip(l, g)]
    m = max(z)
    e = [mpmath.e ** (x - m) for x in z]
    s = sum(e)
    p = [x / s for x in e]
    w = sum(pi * mpmath.mpf(float(qi)) for pi, qi in zip(p, q))
    grad = [float(kappa / tau * pi * (mpmath.mpf(float(qi)) - w)) for pi, qi in zip(p, q)]
    # the scale a float64 sum of the centred terms p_j (q_k - q_j) can resolve
    mass = [float(kappa / tau * pk * sum(pj * abs(mpmath.mpf(float(qk)) - mpmath.mpf(float(qj)))
                                          for pj, qj in zip(p, q))) for pk, qk in zip(p, q)]
    return grad, mass


def test_categorical_gradient_when_saturated():
    grid = np.array([-1.5, -0.5, 0.5, 1.5])
    prob = O.Problem(E=1, R=1, C=4, grid=grid, group=4, H=np.eye(4)[None], noise=False)
    st = O.init_state(prob, np.zeros((1, 4), np.float32), np.arange(1))
    l = np.float32([[[6.0, 0.0, -3.0, 1.0]], [[0.0, 5.0, 0.0, 1.0]], [[-2.0, 0.0, 4.0, 1.0]],
                    [[0.0, -1.0, 0.0, 1.5]]])          # one weight per column, levels down axis 0
    st.logits = l
    tau, kappa = 0.05, 1.0
    fw = O.forward(prob, st, 0, tau, kappa)
    G = np.ones((1, 4))
    dl, _ = O.backward(prob, fw, G, tau, kappa)
    for c in range(4):
        want, mass = _mp_softmax_grad(l[:, 0, c], np.zeros(4), grid, tau, kappa)
        s = float(fw.s[0, c])
        for k in range(4):
            assert abs(dl[k, 0, c] - s * want[k]) <= 1e-12 * abs(s) * mass[k] + 1e-300, (c, k)


def test_binary_gradient_when_saturated():
    for lm, tau in ((9.0, 0.5), (-7.0, 0.25), (0.3, 1.0)):
        p, soft = O.binary_gs(np.array([lm]), np.array([0.0]), O.BINARY_VALUES[0], tau, 1.0)
        got = O.binary_gs_grad(p, soft, O.BINARY_VALUES[0], tau, 1.0)[0]
        # tied logits (-l, l) over the values (0, 1): d/dl of the soft value
        x = 2 * mpmath.mpf(lm) / tau
        p1 = 1 / (1 + mpmath.e ** (-x))
        want = float(2 / mpmath.mpf(tau) * p1 * (1 - p1))
        assert abs(got - want) <= 1e-12 * want, (lm, tau, got, want)
