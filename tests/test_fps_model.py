"""The decision procedure of the GPU draw kernel, modelled on the CPU, against the oracle.

The kernel keeps a pool of the W candidates farthest from the pivots with their exact
distances, and, for every candidate outside the pool, an upper bound of its distance and a
stamp: the number of draws the bound accounts for. A pool candidate is drawn only if it beats
the largest outside bound (ties to the lower index); otherwise that outside candidate is
brought up to date and, if it still leads, drawn. This model replays those decisions in
fp64 and checks that they give exactly the oracle's farthest point sampling for every pool
size, and that each draw refreshes every outside candidate at most once.
"""
import numpy as np
import pytest

import oracle.trevs_oracle as O


def _unit(Z):
    nz = np.sqrt((Z * Z).sum(1))
    return np.divide(Z, nz[:, None], out=np.zeros_like(Z), where=nz[:, None] > 0)


def model_draws(Z, pivots, k_d, pool):
    """(draws, refresh rounds per draw) of the kernel's procedure; `pivots` non-empty."""
    U = _unit(np.asarray(Z, dtype=np.float64))
    n = len(U)
    cand = np.ones(n, dtype=bool)
    dist0 = np.full(n, np.inf)
    for p in pivots:
        cand[p] = False
        dist0 = np.minimum(dist0, 1.0 - U @ U[p])
    ncand = int(cand.sum())
    W = min(pool, ncand, 128)
    order = sorted(np.flatnonzero(cand), key=lambda i: (-dist0[i], i))
    P = sorted(order[:W])
    stamp = np.where(cand, 0, -1)
    ub = dist0.copy()
    for p in P:
        stamp[p] = -1
    pd = {p: dist0[p] for p in P}
    drawn = set()
    draws, rounds = [], []

    def outside():
        live = np.flatnonzero(stamp >= 0)
        return -1 if len(live) == 0 else int(min(live, key=lambda i: (-ub[i], i)))

    o = outside()
    for t in range(k_d):
        r = 0
        while True:
            r += 1
            assert r <= n + 1, "a draw took more rounds than there are candidates"
            avail = [p for p in P if p not in drawn]
            g = min(avail, key=lambda p: (-pd[p], p)) if avail else -1
            if g >= 0 and (o < 0 or (pd[g], -g) > (ub[o], -o)):
                draws.append(g)
                drawn.add(g)
                for p in P:
                    pd[p] = min(pd[p], 1.0 - U[g] @ U[p])
                break
            if stamp[o] == t:
                draws.append(o)
                stamp[o] = -1
                for p in P:
                    if p not in drawn:
                        pd[p] = min(pd[p], 1.0 - U[p] @ U[o])
                o = outside()
                break
            ub[o] = min([ub[o]] + [1.0 - U[o] @ U[draws[k]] for k in range(stamp[o], t)])
            stamp[o] = t
            o = outside()
        rounds.append(r)
    return draws, rounds


def _hypercube(copies, seed):
    v = np.array([[1 - 2 * ((k >> c) & 1) for c in range(6)] for k in range(64)], np.float64)
    Z = np.tile(v, (copies, 1))
    return Z[np.random.default_rng(seed).permutation(len(Z))]


@pytest.mark.parametrize("pool", [1, 2, 5, 17, 64, 128])
def test_model_equals_fps_on_random_rows(pool):
    rng = np.random.default_rng(pool)
    for _ in range(6):
        n = int(rng.integers(20, 160))
        Z = rng.standard_normal((n, 12)) + rng.standard_normal((1, 12)) * rng.uniform(0, 2)
        piv = sorted(rng.choice(n, size=int(rng.integers(1, 10)), replace=False).tolist())
        k_d = int(rng.integers(1, n - len(piv) + 1))
        draws, rounds = model_draws(Z, piv, k_d, pool)
        ref, _ = O.farthest_point_sampling(Z, piv, k_d)
        assert draws == list(ref)
        assert max(rounds) <= n - len(piv) + 1


@pytest.mark.parametrize("pool", [1, 3, 40, 128])
def test_model_equals_fps_with_exact_ties(pool):
    # vertices of {+1, -1}^6, three copies each: every distance is a multiple of 1/3 and
    # duplicates sit at distance 0, so most draws are decided by the lower index
    Z = _hypercube(3, pool)
    piv = [0, 1]
    draws, _ = model_draws(Z, piv, 150, pool)
    ref, _ = O.farthest_point_sampling(Z, piv, 150)
    assert draws == list(ref)


def test_model_with_a_zero_pivot_row():
    rng = np.random.default_rng(3)
    Z = np.vstack([rng.standard_normal((90, 8)), np.zeros((1, 8))])
    piv = [4, 90]                       # row 90 is zero: every distance is capped at 1
    for pool in (1, 8, 128):
        draws, _ = model_draws(Z, piv, 40, pool)
        assert draws == list(O.farthest_point_sampling(Z, piv, 40)[0])


def test_model_row_zero_lead_without_pivots():
    # without pivots the first draw is row 0 and the rest is FPS from it as the one pivot
    rng = np.random.default_rng(5)
    Z = rng.standard_normal((70, 10))
    ref, _ = O.farthest_point_sampling(Z, [], 30)
    draws, _ = model_draws(Z, [0], 29, 20)
    assert [0] + draws == list(ref)
