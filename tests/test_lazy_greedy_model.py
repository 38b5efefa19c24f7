"""The selection's block-lazy rounds pick exactly what the eager greedy of Eq. 4 picks
(CPU model of the scheme, float64; no GPU code involved).

Why the rounds are exact: a candidate's value p_i * rho_i^lambda only shrinks as the basis
grows, so a value computed on an older basis is an upper bound.  A round takes the S
candidates with the largest bounds (the active set), brings their values up to date, and
keeps picking the best active candidate while its exact value beats the largest bound
outside the set (theta): then it beats every candidate's exact value, so it is the eager
argmax.  Keys are (value, lower index first), as in the greedy's tie rule.

The models below share one value function: token i's coordinates on basis vector beta are
computed once, for every token, when beta is added, and its squared residual is its squared
norm minus its coordinates' squares summed in basis order.  A value is then the same number
whenever it is evaluated, so the lazy and the eager runs must agree pick for pick, whatever
S is and whether or not the candidates start from exact values (the projection pass after
R0) or from the bound p_i * ||v_i||^lambda.  The eager model is also held to the oracle."""
import numpy as np
import pytest

from oracle import map_oracle as O


class _Model:
    def __init__(self, p, V, lam, tau):
        self.p, self.V, self.lam, self.tau = p, V, lam, tau
        self.sq = np.einsum("nd,nd->n", V, V)
        self.C = np.zeros((len(p), 0))             # coordinates, one column per basis vector
        self.Q = []

    def value(self, i):
        r2 = self.sq[i]
        for b in range(self.C.shape[1]):
            r2 -= self.C[i, b] ** 2
        if self.lam == 0.0:
            return self.p[i]
        if not (r2 > self.tau * self.sq[i]) or r2 <= 0.0:
            return 0.0
        return self.p[i] * r2 ** (0.5 * self.lam)

    def add(self, j):
        r = self.V[j].copy()
        for q in self.Q:                            # modified Gram-Schmidt on the picked token
            r -= (q @ r) * q
        n2 = r @ r
        if not (n2 > self.tau * self.sq[j]) or n2 <= 0.0:
            return                                  # degenerate: kept, no new direction
        q = r / np.sqrt(n2)
        self.Q.append(q)
        self.C = np.concatenate([self.C, (self.V @ q)[:, None]], axis=1)


def _key(v, i):
    return (v, -i)


def _r0(p, K0):
    return list(np.lexsort((np.arange(len(p)), -p))[:K0])


def eager(p, V, K, K0, lam=1.0, tau=1e-5):
    m = _Model(p, V, lam, tau)
    picks = []
    for j in _r0(p, K0):
        picks.append(int(j))
        m.add(int(j))
    alive = np.ones(len(p), bool)
    alive[picks] = False
    while len(picks) < K:
        cand = np.flatnonzero(alive)
        j = max(cand, key=lambda i: _key(m.value(i), i))
        picks.append(int(j))
        alive[j] = False
        m.add(int(j))
    return picks


def lazy(p, V, K, K0, S, lam=1.0, tau=1e-5, exact_start=True):
    m = _Model(p, V, lam, tau)
    N = len(p)
    picks = []
    for j in _r0(p, K0):
        picks.append(int(j))
        m.add(int(j))
    alive = np.ones(N, bool)
    alive[picks] = False
    if exact_start:                                  # the projection pass: exact values on R0's basis
        U = np.array([m.value(i) for i in range(N)])
    else:                                            # bounds p * ||v||^lambda
        U = p.copy() if lam == 0.0 else p * m.sq ** (0.5 * lam)
    rounds = 0
    while len(picks) < K:
        rounds += 1
        cand = sorted(np.flatnonzero(alive), key=lambda i: _key(U[i], i), reverse=True)
        A, rest = cand[:S], cand[S:]
        theta = _key(U[rest[0]], rest[0]) if rest else None
        for i in A:                                  # the coordinate update
            U[i] = m.value(i)
        while len(picks) < K:
            live = [i for i in A if alive[i]]
            if not live:
                break
            j = max(live, key=lambda i: _key(U[i], i))
            if theta is not None and _key(U[j], j) <= theta:
                break                                # a candidate outside A might be better
            picks.append(int(j))
            alive[j] = False
            m.add(int(j))
            for i in A:
                if alive[i]:
                    U[i] = m.value(i)
        # a round that picks nothing turns S stale bounds into exact values, so at most
        # ceil(N / S) such rounds come before a pick
        assert rounds <= K * (-(-N // S) + 1), "the rounds made no progress"
    lazy.rounds = rounds
    return picks


def _clustered(seed, N=160, D=24, clusters=6, noise=0.3, dup=0):
    rng = np.random.default_rng(seed)
    cent = rng.standard_normal((clusters, D))
    V = cent[rng.integers(clusters, size=N)] + noise * rng.standard_normal((N, D))
    for d in range(dup):                             # exact and near duplicates
        V[N - 1 - d] = V[d] * (1.0 if d % 2 == 0 else 1.0 + 1e-7)
    p = rng.dirichlet(np.full(N, 0.5))
    return p, V


@pytest.mark.parametrize("seed,K,K0,lam", [(0, 24, 12, 1.0), (1, 30, 0, 1.0), (2, 20, 5, 0.5), (3, 16, 8, 2.0),
                                           (4, 40, 20, 1.0), (5, 12, 12, 1.0)])
@pytest.mark.parametrize("S", [1, 2, 5, 16, 64, 1000])
def test_lazy_rounds_pick_like_the_eager_greedy(seed, K, K0, lam, S):
    p, V = _clustered(seed)
    want = eager(p, V, K, K0, lam)
    assert lazy(p, V, K, K0, S, lam, exact_start=True) == want
    assert lazy(p, V, K, K0, S, lam, exact_start=False) == want


@pytest.mark.parametrize("S", [1, 3, 8])
def test_lazy_rounds_with_duplicates_and_degenerate_residuals(S):
    p, V = _clustered(7, dup=6)
    p[:6] += 0.05                                    # the duplicated tokens rank high
    p /= p.sum()
    want = eager(p, V, 30, 4)
    assert lazy(p, V, 30, 4, S) == want
    assert lazy(p, V, 30, 4, S, exact_start=False) == want


@pytest.mark.parametrize("seed,K,K0,lam", [(0, 24, 12, 1.0), (2, 20, 5, 0.5), (3, 16, 8, 2.0), (8, 32, 0, 1.0)])
def test_eager_model_is_the_oracle_greedy(seed, K, K0, lam):
    p, V = _clustered(seed)
    ref = O.select(p, V, K, K0, lam=lam)
    clear = ref["margins"][K0:] > 1e-9              # steps whose order fp64 rounding cannot change
    got = eager(p, V, K, K0, lam)
    assert got[:K0] == ref["picks"][:K0].tolist()
    if clear.all():
        assert got == ref["picks"].tolist()
    else:
        first = K0 + int(np.argmin(clear))
        assert got[:first] == ref["picks"][:first].tolist()


def test_theta_bound_matters():
    # without the theta test a round would keep picking inside a stale active set: with S = 1
    # and exact starts only, the second-best candidate of the first round is never reconsidered
    p, V = _clustered(11)
    want = eager(p, V, 20, 4)

    def no_theta(p, V, K, K0, S):
        m = _Model(p, V, 1.0, 1e-5)
        picks = []
        for j in _r0(p, K0):
            picks.append(int(j))
            m.add(int(j))
        alive = np.ones(len(p), bool)
        alive[picks] = False
        U = np.array([m.value(i) for i in range(len(p))])
        while len(picks) < K:
            A = sorted(np.flatnonzero(alive), key=lambda i: _key(U[i], i), reverse=True)[:S]
            for i in A:
                U[i] = m.value(i)
            j = max(A, key=lambda i: _key(U[i], i))
            picks.append(int(j))
            alive[j] = False
            m.add(int(j))
            U[j] = -1.0
        return picks

    assert any(no_theta(p, V, 20, 4, S) != want for S in (1, 2, 3))
