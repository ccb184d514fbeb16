"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a closed
form, an identity or bound the paper proves, brute force on a tiny input, a
textbook special case, or a hand-worked example.  None of them re-types the
oracle's own formula.
"""

import itertools
import math

import numpy as np
import pytest
from scipy.special import softmax as sp_softmax

from oracle import gmc_oracle as O

P = O.params()


def rng(seed=0):
    return np.random.default_rng(seed)


# --------------------------------------------------------------------------
# a1 budget: Sec. 3.1 and the totality rule
# --------------------------------------------------------------------------
def test_budget_totality():
    assert O.budget(16, 64) == 16
    assert O.budget(100, 64) == 64          # K_r > N clamps to N
    assert O.budget(0, 64) == 1             # at least one carrier per image
    assert O.budget(2, 64, n_images=3) == 3  # K_r < I expands to I


# --------------------------------------------------------------------------
# a2 native message slice: Eq. (cond-native-message)
# --------------------------------------------------------------------------
def _slice_case(N=6, T=3, H=4, Hkv=2, d=8, seed=1):
    r = rng(seed)
    Q = r.standard_normal((T, H, d))
    K = r.standard_normal((N + T, Hkv, d))
    return Q, K


def test_message_slice_brute_force_loops():
    """Element-wise python loops with math.exp on a tiny case."""
    N, T, H, Hkv, d = 5, 3, 4, 2, 4
    Q, K = _slice_case(N, T, H, Hkv, d, seed=2)
    A = O.message_slice(Q, K, N)
    for h in range(H):
        g = h // 2
        for t in range(T):
            keys = list(range(N)) + [N + k for k in range(t + 1)]
            sc = [sum(Q[t, h, c] * K[k, g, c] for c in range(d)) / math.sqrt(d) for k in keys]
            den = sum(math.exp(s) for s in sc)
            for i in range(N):
                assert A[h, t, i] == pytest.approx(math.exp(sc[i]) / den, rel=1e-12)


def test_message_slice_native_mass_and_causality():
    N, T = 6, 4
    Q, K = _slice_case(N, T)
    A = O.message_slice(Q, K, N)
    # The visual slice is not renormalised: the text keys take part of the mass.
    vis = A.sum(axis=2)
    assert np.all(vis < 1.0) and np.all(vis > 0.0)
    # scipy softmax over the masked score row reproduces the visual columns.
    h, t = 3, 2
    g = h // 2
    s = Q[t, h] @ K[: N + t + 1, g].T / math.sqrt(Q.shape[2])
    np.testing.assert_allclose(A[h, t], sp_softmax(s)[:N], rtol=1e-12)
    # A future text key (position > N+t) never changes row t.
    K2 = K.copy()
    K2[N + 3] += 100.0
    A2 = O.message_slice(Q, K2, N)
    np.testing.assert_array_equal(A2[:, :3], A[:, :3])
    assert not np.allclose(A2[:, 3], A[:, 3])


def test_message_slice_text_key_dominates():
    """A text key aligned with the query takes almost all mass (visual-only renorm would give 1)."""
    N, T, H, d = 4, 1, 1, 4
    Q = np.zeros((T, H, d)); Q[0, 0, 0] = 10.0
    K = np.zeros((N + T, 1, d)); K[N, 0, 0] = 10.0
    A = O.message_slice(Q, K, N)
    # scores: visual 0, text 100/2 = 50  ->  visual mass 4 / (4 + e^50)
    assert A.sum() == pytest.approx(4.0 / (4.0 + math.exp(50.0)), rel=1e-12)


def test_message_slice_single_query_is_plain_softmax():
    N, T, H, d = 7, 1, 1, 16
    r = rng(3)
    Q = r.standard_normal((T, H, d)); K = r.standard_normal((N + T, 1, d))
    A = O.message_slice(Q, K, N)
    ref = sp_softmax(K[:, 0] @ Q[0, 0] / 4.0)
    np.testing.assert_allclose(A[0, 0], ref[:N], rtol=1e-12)


# --------------------------------------------------------------------------
# a3/a4 probe, mass coordinate, grounded clients: Eq. (1), (2)
# --------------------------------------------------------------------------
def test_mass_coordinate_floor_gives_attention_proportional_clients():
    """V = 0: Z = 0, sigma = eps_mass, so ||u|| = A * 1e-8 and P^G = A / sum A."""
    N, T, H, d = 5, 2, 2, 4
    Q, K = _slice_case(N, T, H, 1, d, seed=4)
    A = O.message_slice(Q, K, N)
    Z, sigma = O.probe_values(np.zeros((N, 1, d)), rng(5).standard_normal((H, d, 4)), H, P)
    assert np.all(sigma == 1e-8)
    PG, act = O.grounded_clients(O.atom_norms(A, Z, sigma))
    assert act.all()
    np.testing.assert_allclose(PG, A / A.sum(axis=2, keepdims=True), rtol=1e-12)


def test_mass_coordinate_closed_form_and_rotation_invariance():
    N, H, Hkv, d = 9, 4, 2, 8
    r = rng(6)
    V = r.standard_normal((N, Hkv, d))
    W = r.standard_normal((H, d, 4))
    Z, sigma = O.probe_values(V, W, H, P)
    for h in range(H):
        brute = sum((V[i, h // 2] @ W[h][:, c]) ** 2 for i in range(N) for c in range(4))
        assert sigma[h] == pytest.approx(math.sqrt(brute / (N * 4)), rel=1e-12)
    # Rotating the probe inside its span (P -> P Rot) leaves ||Z_h[i]|| and sigma unchanged.
    Rot, _ = np.linalg.qr(r.standard_normal((4, 4)))
    Z2, s2 = O.probe_values(V, W @ Rot, H, P)
    np.testing.assert_allclose(np.linalg.norm(Z2, axis=2), np.linalg.norm(Z, axis=2), rtol=1e-12)
    np.testing.assert_allclose(s2, sigma, rtol=1e-12)


def test_orthonormal_probe():
    G = rng(7).standard_normal((64, 4))
    Pm = O.orthonormal_probe(G)
    np.testing.assert_allclose(Pm.T @ Pm, np.eye(4), atol=1e-12)
    # span(P) = span(G): projecting G onto P reproduces G.
    np.testing.assert_allclose(Pm @ (Pm.T @ G), G, atol=1e-12)


def test_grounded_client_hand_example():
    """A = [.5, .25, .25], ||[Z;sigma]|| = [1, 2, 2] -> ||u|| = [.5, .5, .5] -> P^G = 1/3 each."""
    A = np.array([[[0.5, 0.25, 0.25]]])
    Z = np.array([[[1.0, 0, 0, 0], [0, 2.0, 0, 0], [0, 0, 0, 2.0]]]) * 1.0
    sigma = np.array([0.0])
    un = O.atom_norms(A, Z, sigma)
    np.testing.assert_allclose(un, [[[0.5, 0.5, 0.5]]])
    PG, act = O.grounded_clients(un)
    np.testing.assert_allclose(PG, [[[1 / 3, 1 / 3, 1 / 3]]])
    assert act.all()


def test_zero_energy_row_is_inactive():
    un = np.zeros((1, 2, 3)); un[0, 1] = [1.0, 3.0, 0.0]
    PG, act = O.grounded_clients(un)
    assert act.tolist() == [[False, True]]
    assert PG[0, 0].sum() == 0.0
    np.testing.assert_allclose(PG[0, 1], [0.25, 0.75, 0.0])


# --------------------------------------------------------------------------
# a5 query weights, head clusters, energy: Eq. (cond-head-pattern), (cond-head-weight),
#    (cond-grounded-energy)
# --------------------------------------------------------------------------
def test_query_weights_terminal_double():
    np.testing.assert_allclose(O.query_weights(4, P), [0.2, 0.2, 0.2, 0.4])
    np.testing.assert_allclose(O.query_weights(1, P), [1.0])


def _heads_with_patterns(blocks, N=8, T=2):
    """Heads whose attention lives on disjoint token blocks; heads in one block are identical."""
    H = len(blocks)
    A = np.zeros((H, T, N))
    for h, blk in enumerate(blocks):
        A[h, :, blk] = 1.0 / len(blk)
    Z = np.ones((H, N, 4))
    sigma = np.ones(H)
    return A, Z, sigma


def test_identical_heads_form_one_cluster_with_uniform_weights():
    A, Z, s = _heads_with_patterns([[0, 1, 2]] * 5)
    hc = O.head_clusters(A, Z, s, P)
    assert hc.n_clusters == 1
    np.testing.assert_allclose(hc.omega, np.full(5, 0.2))
    np.testing.assert_allclose(hc.dispersion, 0.0, atol=1e-12)


def test_orthogonal_head_families_get_equal_cluster_mass():
    # family sizes 3, 1, 2, 1 on disjoint blocks -> 4 clusters of mass 1/4 each
    fam = [[0, 1]] * 3 + [[2, 3]] + [[4, 5]] * 2 + [[6, 7]]
    A, Z, s = _heads_with_patterns(fam)
    hc = O.head_clusters(A, Z, s, P)
    assert hc.n_clusters == 4
    np.testing.assert_allclose(hc.omega, [1 / 12] * 3 + [1 / 4] + [1 / 8] * 2 + [1 / 4])
    assert hc.omega.sum() == pytest.approx(1.0)
    # the specialised single heads (3 and 6) weigh as much as a whole family
    assert hc.omega[3] == pytest.approx(hc.omega[:3].sum())


def test_farthest_first_hand_example():
    """Patterns e0, e1, (e0+e1)/sqrt2, e2 with head 2 the largest: centres 2, 3, 0, 1.

    pre-norms are equal after the unit-mean-norm scaling except for the count of
    atoms; cosines: c(0,1)=0, c(0,2)=c(1,2)=1/sqrt2, c(3,.)=0.  First centre is
    the largest pre-normalisation pattern (all tie -> lowest index 0); then the
    head with the smallest max-cosine to {0}: head 1 or 3 (both 0) -> 1; then
    to {0,1}: head 3 (0 < 1/sqrt2) ; then head 2.
    """
    N, T = 3, 1
    A = np.zeros((4, T, N))
    A[0, 0] = [1, 0, 0]
    A[1, 0] = [0, 1, 0]
    A[2, 0] = [0.5, 0.5, 0]
    A[3, 0] = [0, 0, 1]
    Z = np.zeros((4, N, 4))
    sigma = np.ones(4)
    hc = O.head_clusters(A, Z, sigma, P)
    assert hc.cos[0, 2] == pytest.approx(1 / math.sqrt(2))
    assert hc.centres == [0, 1, 3, 2]
    assert hc.n_clusters == 4


def test_head_weight_inverse_dispersion():
    """Eq. (cond-head-weight) by hand: one cluster of two heads with d = (0.05, 0.15)."""
    # patterns u0 = e0, u1 = (cos a) e0 + (sin a) e1 with the mean direction mu at a/2:
    # d_h = 1 - cos(a/2) for both -> equal weights 1/2.
    N, T = 2, 1
    a = 0.3
    A = np.zeros((2, T, N)); Z = np.zeros((2, N, 4)); sigma = np.ones(2)
    A[0, 0] = [1.0, 0.0]
    A[1, 0] = [math.cos(a), math.sin(a)]
    p = O.params(max_head_clusters=1)
    hc = O.head_clusters(A, Z, sigma, p)
    np.testing.assert_allclose(hc.dispersion, [1 - math.cos(a / 2)] * 2, rtol=1e-9)
    np.testing.assert_allclose(hc.omega, [0.5, 0.5])
    # three heads, two identical: mu tilts toward the pair, so the pair weighs more
    A3 = np.zeros((3, T, N)); Z3 = np.zeros((3, N, 4))
    A3[0, 0] = [1.0, 0.0]; A3[1, 0] = [1.0, 0.0]; A3[2, 0] = [math.cos(a), math.sin(a)]
    hc3 = O.head_clusters(A3, Z3, np.ones(3), p)
    mu = np.array([2 + math.cos(a), math.sin(a)]); mu /= np.linalg.norm(mu)
    d = np.array([1 - mu[0], 1 - mu[0], 1 - (math.cos(a) * mu[0] + math.sin(a) * mu[1])])
    w = 1 / (d + 0.05)
    np.testing.assert_allclose(hc3.omega, w / w.sum(), rtol=1e-9)


def test_energy_closed_form_and_fallback():
    # one head (omega = 1), two queries with nu = [1/3, 2/3]
    un = np.array([[[3.0, 0.0], [0.0, 6.0]]])
    nu = O.query_weights(2, P)
    e, eb = O.message_energy(un, np.array([1.0]), nu)
    np.testing.assert_allclose(e, [math.sqrt(9 / 3), math.sqrt(36 * 2 / 3)])
    np.testing.assert_allclose(eb.mean(), 1.0)
    e0, eb0 = O.message_energy(np.zeros((1, 2, 3)), np.array([1.0]), nu)
    np.testing.assert_array_equal(eb0, np.ones(3))


# --------------------------------------------------------------------------
# a6/a7 appearance and spatial banks: Eq. (cond-aux-clients), (cond-gibbs)
# --------------------------------------------------------------------------
def test_appearance_gibbs_modal_ratio():
    """P^V_m(j)/P^V_m(m) = exp(-||x_m - x_j||^2 / (2 tau_v)) (Eq. (cond-gibbs))."""
    h = rng(8).standard_normal((12, 32)) * rng(9).uniform(0.5, 3, size=(12, 1))
    cos = O.cosine_matrix(h, P)
    PV = O.appearance_clients(cos, P)
    np.testing.assert_allclose(PV.sum(axis=1), 1.0, rtol=1e-12)
    x = h / np.linalg.norm(h, axis=1, keepdims=True)
    for m in range(12):
        for j in range(12):
            ratio = math.exp(-np.sum((x[m] - x[j]) ** 2) / (2 * 0.2))
            assert PV[m, j] / PV[m, m] == pytest.approx(ratio, rel=1e-10)


def test_spatial_bank_on_landmark_grid():
    """On a 16x16 grid the token coordinates coincide with the landmarks."""
    PS = O.spatial_clients(16, 16, P)
    assert PS.shape == (256, 256)
    np.testing.assert_allclose(PS.sum(axis=1), 1.0, rtol=1e-12)
    assert np.all(np.argmax(PS, axis=1) == np.arange(256))
    # neighbour one cell right: distance 1/16 -> ratio exp(-(1/16)^2 / 0.02)
    assert PS[0, 1] / PS[0, 0] == pytest.approx(math.exp(-(1 / 16) ** 2 / 0.02), rel=1e-12)
    # diagonal neighbour: distance^2 = 2/256
    assert PS[17, 0] / PS[17, 17] == pytest.approx(math.exp(-(2 / 256) / 0.02), rel=1e-12)


def test_spatial_coordinates_are_normalised_centres():
    g = O.grid_coords(2, 4)
    np.testing.assert_allclose(g[5], [0.75, 0.375])   # i = 1*4 + 1
    lm = O.landmark_coords(16)
    np.testing.assert_allclose(lm[17], [1.5 / 16, 1.5 / 16])


def _tiny_result(seed=0, **kw):
    from paper_2608_02134_gb300 import workloads
    wl = workloads.make("tiny", **kw)
    im = wl.image(0)
    res = O.compress(im.hidden.astype(np.float64), im.keys.astype(np.float64),
                     im.values.astype(np.float64), im.queries.astype(np.float64),
                     im.pos, wl.probe().astype(np.float64), wl.gh, wl.gw, wl.K)
    return wl, im, res


def test_bank_masses_and_effective_shares():
    """Rows sum to beta_b / M_b; Z_b = F_b(V) matches Eq. (cond-effective-bank-mass)."""
    wl, im, res = _tiny_result()
    cm = res.clients
    G, V, S = (cm.C[cm.banks[b]] for b in ("grounded", "appearance", "spatial"))
    assert G.sum() == pytest.approx(0.5, rel=1e-12)     # sum_h omega_h sum_t nu_t = 1
    np.testing.assert_allclose(V.sum(axis=1), 0.5 / wl.N, rtol=1e-12)
    np.testing.assert_allclose(S.sum(axis=1), 0.25 / 256, rtol=1e-12)
    sat = O.bank_saturation(cm, range(wl.N))
    PV = O.appearance_clients(res.cos, P)
    assert sat["appearance"][1] == pytest.approx(0.5 / wl.N * PV.max(axis=1).sum(), rel=1e-12)
    assert sum(v[2] for v in sat.values()) == pytest.approx(1.0)


def test_grounded_row_masses_follow_head_and_query_weights():
    """Row (h, t) carries beta_G * omega_h * nu_t: the terminal query row of a head weighs
    twice any other row of that head, and a head's rows together carry beta_G * omega_h."""
    wl, im, res = _tiny_result()
    T = wl.T[0]
    G = res.clients.C[res.clients.banks["grounded"]].reshape(wl.H, T, wl.N).sum(axis=2)
    for h in range(wl.H):
        np.testing.assert_allclose(G[h, T - 1] / G[h, :T - 1], 2.0, rtol=1e-12)
        assert G[h].sum() == pytest.approx(0.5 * res.heads.omega[h], rel=1e-12)


def test_coverage_to_quantization_bound():
    """Eq. (7) / (cond-coverage-quantization) on random supports."""
    h = rng(10).standard_normal((40, 16))
    cos = O.cosine_matrix(h, P)
    PV = O.appearance_clients(cos, P)
    x = h / np.linalg.norm(h, axis=1, keepdims=True)
    N = 40
    for seed in range(5):
        S = rng(100 + seed).choice(N, size=8, replace=False)
        d2 = np.array([min(np.sum((x[m] - x[j]) ** 2) for j in S) for m in range(N)])
        r = PV[:, S].max(axis=1) / np.diag(PV)
        DV = 0.5 / N * np.sum(np.diag(PV) * (1 - r))
        p0, r0 = np.diag(PV).min(), r.min()
        assert d2.mean() <= 2 * 0.2 / (0.5 * p0 * r0) * DV + 1e-15
        # exact identity inside the proof: r_m = exp(-d_m^2 / (2 tau_v))
        np.testing.assert_allclose(r, np.exp(-d2 / 0.4), rtol=1e-10)


# --------------------------------------------------------------------------
# a8 selection: Eq. (3), (4), (6); Eq. (cond-submodular), (cond-batched-bound),
#    (cond-final-cert)
# --------------------------------------------------------------------------
def _rand_C(M, N, seed):
    r = rng(seed)
    C = r.exponential(size=(M, N)) * (r.uniform(size=(M, N)) < 0.6)
    return C / C.sum()


def test_facility_normalised_monotone_submodular_brute_force():
    C = _rand_C(7, 6, 11)
    assert O.facility_value(C, []) == 0.0
    subsets = [s for k in range(7) for s in itertools.combinations(range(6), k)]
    F = {s: O.facility_value(C, s) for s in subsets}
    for A_ in subsets:
        for B_ in subsets:
            if set(A_) <= set(B_):
                assert F[A_] <= F[B_] + 1e-15
                for i in set(range(6)) - set(B_):
                    gA = O.facility_value(C, A_ + (i,)) - F[A_]
                    gB = O.facility_value(C, B_ + (i,)) - F[B_]
                    assert gA >= gB - 1e-15


@pytest.mark.parametrize("seed", range(6))
def test_batched_certificate_and_greedy_bound_vs_brute_force(seed):
    N, K = 12, 4
    C = _rand_C(15, N, 20 + seed)
    p = O.params(batch_b=2, pool_mult=2)
    best = max(O.facility_value(C, s) for s in itertools.combinations(range(N), K))
    sel = O.select_support(C, K, p)
    FS = O.facility_value(C, sel.order)
    cB = O.batched_certificate(sel)
    assert 0.0 <= cB <= 1.0
    assert FS >= cB * best - 1e-15                       # Eq. (6) with F(S_0) = 0
    assert FS / O.facility_value(C, range(N)) <= FS / best + 1e-15 <= 1.0 + 1e-15
    g = O.select_support(C, K, p, mode="greedy")
    assert O.facility_value(C, g.order) >= (1 - (1 - 1 / K) ** K) * best - 1e-15
    # greedy recovers the first element of the exact greedy chain: argmax column sum
    assert g.order[0] == int(np.argmax(C.sum(axis=0)))


def test_selection_exact_cardinality_unique_and_in_range():
    C = _rand_C(50, 40, 30)
    sel = O.select_support(C, 23, P)
    assert len(sel.order) == 23 and len(set(sel.order)) == 23
    assert min(sel.order) >= 0 and max(sel.order) < 40
    # round sizes: full batches of 16 while gains are positive
    assert [len(r.batch) for r in sel.rounds] == [16, 7]


def test_zero_gain_fill_in_index_order_keeps_F():
    """Identical tokens: after the first batch every gain is zero and the fill is 16..K-1."""
    col = rng(31).exponential(size=(9, 1))
    C = np.repeat(col, 30, axis=1)
    sel = O.select_support(C, 20, P)
    assert sel.order == list(range(20))
    assert sel.rounds[1].fill and sel.rounds[1].batch.tolist() == list(range(16, 20))
    assert sel.rounds[1].F_after == sel.rounds[1].F_before


def test_responsibility_round_hand_example():
    """One round of Eq. (4) worked by hand (tests/golden/responsibility_round.txt)."""
    from tests.golden_cases import load_case
    case = load_case("responsibility_round.txt")
    C = np.array(case["C"])
    p = O.params(batch_b=int(case["b"]), pool_mult=int(case["pool_mult"]))
    sel = O.select_support(C, int(case["K"]), p)
    r0 = sel.rounds[0]
    np.testing.assert_allclose(r0.gains, case["u"], rtol=1e-12)
    assert r0.pool.tolist() == case["pool"]
    np.testing.assert_allclose(r0.scores, case["s"], rtol=1e-9)
    assert r0.batch.tolist() == case["batch"]


def test_selection_trivial_cases():
    C = _rand_C(6, 5, 40)
    sel = O.select_support(C, 5, P)
    assert sorted(sel.order) == [0, 1, 2, 3, 4]
    sel1 = O.select_support(C, 1, P)
    assert len(sel1.order) == 1


# --------------------------------------------------------------------------
# a9 assignment: Eq. (cond-assignment), (cond-population-gate), (cond-assignment-bound)
# --------------------------------------------------------------------------
def test_assignment_without_gate_is_cosine_nearest_neighbour():
    h = rng(50).standard_normal((36, 8))
    cos = O.cosine_matrix(h, P)
    S = np.array([1, 7, 20, 33])
    p = O.params(gate_scale=1e9)           # s_x = 0
    a = O.assign_population(cos, S, 6, 6, p)
    assert a.s_x == 0.0
    x = h / np.linalg.norm(h, axis=1, keepdims=True)
    for i in range(36):
        want = i if i in S else S[int(np.argmin([np.sum((x[i] - x[j]) ** 2) for j in S]))]
        assert a.pi[i] == want


def test_assignment_gap_gate_closed_form_and_bound():
    h = rng(51).standard_normal((64, 8))
    cos = O.cosine_matrix(h, P)
    S = np.array([0, 9, 27, 40, 63])
    a = O.assign_population(cos, S, 8, 8, P)
    disc = [i for i in range(64) if i not in S]
    gaps = []
    for i in disc:
        v = sorted(cos[i, S], reverse=True)
        gaps.append(v[0] - v[1])
    assert a.delta_bar == pytest.approx(np.mean(gaps), rel=1e-12)
    assert a.s_x == pytest.approx(1 - math.exp(-(np.mean(gaps) / 0.08) ** 8), rel=1e-12)
    assert all(a.pi[j] == j for j in S)
    # Eq. (cond-assignment-bound): ||x_i - x_pi(i)||^2 <= d_i(S)^2 + 2 lambda_i, lambda_i = 0.5 s_x g_i
    x = h / np.linalg.norm(h, axis=1, keepdims=True)
    for i in disc:
        d2 = min(np.sum((x[i] - x[j]) ** 2) for j in S)
        lam = 0.5 * a.s_x * a.g[i]
        assert np.sum((x[i] - x[a.pi[i]]) ** 2) <= d2 + 2 * lam + 1e-12


def test_assignment_single_representative_and_no_discard():
    h = rng(52).standard_normal((9, 4))
    cos = O.cosine_matrix(h, P)
    a = O.assign_population(cos, np.array([4]), 3, 3, P)
    assert np.all(a.pi == 4) and np.all(a.delta == 0) and a.s_x == 0.0
    b = O.assign_population(cos, np.arange(9), 3, 3, P)
    assert b.delta_bar == 0.0 and b.s_x == 0.0 and np.all(b.pi == np.arange(9))


def test_assignment_spatial_gate_hand_example():
    """Eq. (cond-assignment) and (cond-population-gate) worked by hand
    (tests/golden/assignment_spatial_gate.txt): the spatial term, its gate and
    the grid coordinates each decide one token's representative."""
    from tests.golden_cases import load_case
    c = load_case("assignment_spatial_gate.txt")
    N = c["gh"] * c["gw"]
    S = np.array(c["S"])
    cos = np.eye(N)
    for i, row in c["cos_to_S"].items():
        cos[int(i), S] = row
        cos[S, int(i)] = row
    a = O.assign_population(cos, S, c["gh"], c["gw"], P)
    assert a.delta_bar == pytest.approx(c["delta_bar"], rel=1e-12)
    assert a.s_x == pytest.approx(c["s_x"], rel=1e-12)
    for i, g in c["g"].items():
        assert a.g[int(i)] == pytest.approx(g, rel=1e-10)
    for i, kap in c["kappa"].items():
        assert a.kappa_best[int(i)] == pytest.approx(max(kap), rel=1e-12)
        assert a.kappa_chosen[int(i)] == pytest.approx(max(kap), rel=1e-12)
    assert a.pi.tolist() == c["pi"]


def test_population_weights_and_transport_hand_example():
    """Eq. (cond-grounded-energy), (cond-population-gate) and (cond-transport)
    worked by hand (tests/golden/population_transport.txt) at s_x = 1 - 1/e."""
    from tests.golden_cases import load_case
    c = load_case("population_transport.txt")
    e = np.array(c["energy"])
    e_o, ebar = O.message_energy(e[None, None, :], np.ones(1), np.ones(1))
    np.testing.assert_allclose(e_o, e, rtol=1e-15)
    np.testing.assert_allclose(ebar, c["ebar"], rtol=1e-15)
    np.testing.assert_allclose(O.population_weights(ebar, c["s_x"], P), c["m"], rtol=1e-14)
    tr = O.transport(np.array(c["h"]), np.array(c["S"]), np.array(c["pi"]),
                     np.array(c["m_transport"]), P)
    np.testing.assert_allclose(tr.mass, c["M"], rtol=1e-15)
    np.testing.assert_allclose(tr.centroid, c["centroid"], rtol=1e-15, atol=1e-15)
    np.testing.assert_allclose(tr.restored, c["restored"], rtol=1e-13, atol=1e-15)


# --------------------------------------------------------------------------
# a10 transport: Eq. (5), (cond-population-moment), (cond-centroid-optimum), (cond-rms-bound)
# --------------------------------------------------------------------------
def _transport_case(seed=60, N=30, D=12, K=5):
    r = rng(seed)
    h = r.standard_normal((N, D)) * r.uniform(0.5, 2, size=(N, 1))
    S = np.sort(r.choice(N, size=K, replace=False))
    pi = S[r.integers(0, K, size=N)]
    pi[S] = S
    m = O.population_weights(r.uniform(0, 3, size=N), 0.7, P)
    return h, S, pi, m


def test_transport_conserves_mass_and_first_moment():
    h, S, pi, m = _transport_case()
    tr = O.transport(h, S, pi, m, P)
    assert tr.mass.sum() == pytest.approx(m.sum(), rel=1e-13)
    np.testing.assert_allclose((tr.mass[:, None] * tr.centroid).sum(0), (m[:, None] * h).sum(0),
                               rtol=1e-12, atol=1e-12)
    W = rng(61).standard_normal((7, h.shape[1]))
    np.testing.assert_allclose((tr.mass[:, None] * (tr.centroid @ W.T)).sum(0),
                               (m[:, None] * (h @ W.T)).sum(0), rtol=1e-11, atol=1e-11)


def test_population_weights_positive():
    eb = rng(62).uniform(0, 5, size=100)
    for sx in (0.0, 0.3, 1.0):
        assert np.all(O.population_weights(eb, sx, P) >= 0.5)
    np.testing.assert_array_equal(O.population_weights(eb, 0.0, P), np.ones(100))


def test_centroid_optimality_identity():
    h, S, pi, m = _transport_case(63)
    tr = O.transport(h, S, pi, m, P)
    u = rng(64).standard_normal(h.shape[1])
    for k, j in enumerate(S):
        mem = np.flatnonzero(pi == j)
        E = lambda v: float(np.sum(m[mem] * np.sum((h[mem] - v) ** 2, axis=1)))
        assert E(u) == pytest.approx(E(tr.centroid[k]) + tr.mass[k] * np.sum((u - tr.centroid[k]) ** 2),
                                     rel=1e-12)


def test_rms_restoration_singleton_and_scale():
    h, S, pi, m = _transport_case(65)
    pi = pi.copy()
    pi[pi == S[0]] = S[1]
    pi[S[0]] = S[0]                     # S[0] alone in its cluster
    tr = O.transport(h, S, pi, m, P)
    r0 = np.sqrt(np.mean(h[S[0]] ** 2))
    np.testing.assert_allclose(tr.restored[0], h[S[0]] * r0 / (r0 + 1e-6), rtol=1e-12)
    rr = np.sqrt(np.mean(tr.restored ** 2, axis=1))
    rh = np.sqrt(np.mean(h[S] ** 2, axis=1))
    np.testing.assert_allclose(rr, rh, rtol=1e-5)
    # Eq. (cond-rms-bound) with beta = 1
    Epre = sum(m[i] * np.sum((h[i] - tr.centroid[list(S).index(pi[i])]) ** 2) for i in range(len(h)))
    Epost = sum(m[i] * np.sum((h[i] - tr.restored[list(S).index(pi[i])]) ** 2) for i in range(len(h)))
    zeta2 = np.sum((tr.restored - tr.centroid) ** 2, axis=1)
    assert Epost <= 2 * Epre + 2 * np.sum(tr.mass * zeta2) + 1e-9


# --------------------------------------------------------------------------
# whole step on the tiny workload: Algorithm 1 steps 2-6 and the numerical checks
# --------------------------------------------------------------------------
def test_tiny_end_to_end_invariants():
    wl, im, res = _tiny_result()
    N, T, K = wl.N, wl.T[0], wl.K
    S = res.support
    assert S.size == K and np.all(np.diff(S) > 0) and S[0] >= 0 and S[-1] < N
    assert np.all(res.assignment.pi[S] == S)
    assert np.all(res.transport.mass > 0)
    assert np.all(np.isfinite(res.out_hidden))
    np.testing.assert_array_equal(res.out_hidden[K:], im.hidden[N:])          # text rows unchanged
    np.testing.assert_array_equal(res.out_pos, im.pos[:, np.r_[S, N + np.arange(T)]])
    np.testing.assert_array_equal(res.out_kv[0, :K], im.keys[S])
    np.testing.assert_array_equal(res.out_kv[1, K:], im.values[N:])
    assert res.out_hidden.shape == (K + T, wl.D)


def test_identity_when_K_equals_N():
    wl, im, res = _tiny_result(K=64)
    assert res.identity
    np.testing.assert_array_equal(res.out_hidden, im.hidden)
    np.testing.assert_array_equal(res.out_pos, im.pos)
    wl2, im2, res2 = _tiny_result(K=1000)
    assert res2.identity and res2.K == 64


# --------------------------------------------------------------------------
# direct pins of the helper steps (each also runs inside the steps above)
# --------------------------------------------------------------------------
def test_head_patterns_hand_example_and_scale_invariance():
    # Eq. (cond-head-pattern): atoms u_i^{h,t} = A[h,t,i] [Z_h[i]; sigma_h],
    # divided by their mean norm over all (t, i).
    # head 0: one atom [3, 4] (norm 5) and a zero atom -> mean norm 2.5,
    #         U_0 = [1.2, 1.6, 0, 0], ||U_0|| = 2;
    # head 1: atoms [0, 0.5] twice -> mean norm 0.5, U_1 = [0, 1, 0, 1], ||U_1|| = sqrt 2;
    # head 2: no attention -> the zero pattern.
    A = np.array([[[1.0, 0.0]], [[0.5, 0.5]], [[0.0, 0.0]]])
    Z = np.array([[[3.0], [0.0]], [[0.0], [0.0]], [[1.0], [1.0]]])
    sigma = np.array([4.0, 1.0, 1.0])
    cos, pre, _ = O.head_patterns(A, Z, sigma)
    np.testing.assert_allclose(pre, [2.0, math.sqrt(2.0), 0.0], atol=1e-15)
    np.testing.assert_allclose(cos[0, 1], 1.6 / (2.0 * math.sqrt(2.0)), rtol=1e-14)
    np.testing.assert_allclose(np.diag(cos)[:2], [1.0, 1.0], rtol=1e-14)
    assert cos[2, 2] == 0.0 and cos[0, 2] == 0.0
    # the mean-norm normalisation makes a pattern blind to the scale of A_h
    A2 = A.copy()
    A2[0] *= 7.0
    cos2, pre2, _ = O.head_patterns(A2, Z, sigma)
    np.testing.assert_allclose(cos2, cos, rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(pre2, pre, rtol=1e-13, atol=1e-15)


def test_client_matrix_row_masses_and_layout():
    # Eq. (cond-coverage): every active row of a bank carries its bank's mass;
    # the client matrix stacks grounded rows (h, t) h-major, appearance rows,
    # then the landmark rows.
    H, T, N, L = 2, 3, 5, 4
    g = rng(3)
    PG = g.random((H, T, N))
    PG /= PG.sum(axis=2, keepdims=True)
    active = np.ones((H, T), dtype=bool)
    active[1, 2] = False
    PG[1, 2] = 0.0
    omega = np.array([0.25, 0.75])
    nu = O.query_weights(T, P)
    PV = g.random((N, N))
    PV /= PV.sum(axis=1, keepdims=True)
    PS = g.random((L, N))
    PS /= PS.sum(axis=1, keepdims=True)
    cm = O.client_matrix(PG, active, omega, nu, PV, PS, P)
    assert cm.C.shape == (H * T + N + L, N)
    rows = cm.C.sum(axis=1)
    for h in range(H):
        for t in range(T):
            want = P["beta_G"] * omega[h] * nu[t] if active[h, t] else 0.0
            assert rows[h * T + t] == pytest.approx(want, rel=1e-13, abs=1e-15)
    np.testing.assert_allclose(rows[H * T:H * T + N], P["beta_V"] / N, rtol=1e-13)
    np.testing.assert_allclose(rows[H * T + N:], P["beta_S"] / L, rtol=1e-13)
    # grounded row (1, 0) is P^G_{1,0} scaled, column for column
    np.testing.assert_allclose(cm.C[1 * T + 0] / rows[1 * T + 0], PG[1, 0], rtol=1e-13)


def test_stable_top_matches_brute_force_with_ties():
    g = rng(4)
    for _ in range(50):
        n = int(g.integers(1, 12))
        vals = g.integers(0, 4, n).astype(float)   # many ties
        ids = g.permutation(100)[:n]
        k = int(g.integers(0, n + 1))
        pairs = sorted(zip(vals, ids), key=lambda x: (-x[0], x[1]))
        want = [int(i) for _, i in pairs[:k]]
        assert [int(i) for i in O.stable_top(vals, ids, k)] == want


def test_rms_and_unit_states_closed_forms():
    assert O.rms(np.array([3.0, 4.0])) == pytest.approx(math.sqrt(12.5), rel=1e-15)
    assert O.rms(np.full(7, -2.5)) == pytest.approx(2.5, rel=1e-15)
    h = np.array([[3.0, 4.0, 0.0], [0.0, 0.0, 0.0], [1e-3, 0.0, 0.0]])
    x = O.unit_states(h, P)
    np.testing.assert_allclose(x[0], [0.6, 0.8, 0.0], rtol=1e-15)
    np.testing.assert_array_equal(x[1], 0.0)                     # eps keeps a zero row zero
    np.testing.assert_allclose(x[2], [1.0, 0.0, 0.0], rtol=1e-15)
    # cosines of scaled states are those of the states
    np.testing.assert_allclose(O.cosine_matrix(5.0 * h, P), O.cosine_matrix(h, P), rtol=1e-14)


def test_compaction_rows_index_map():
    # Appendix "Index map and physical token accounting": kept visual rows in
    # ascending source order, then every text row, K + T rows in all.
    rows = O.compaction_rows(np.array([1, 4, 6]), N=8, T=3)
    np.testing.assert_array_equal(rows, [1, 4, 6, 8, 9, 10])
    assert O.compaction_rows(np.array([], dtype=np.int64), N=4, T=0).size == 0


# --------------------------------------------------------------------------
# historical message views (Appendix "Native message clients": every view is a
# separate client collection; Eq. (cond-head-pattern) concatenates the views)
# --------------------------------------------------------------------------
def _tiny_with_history(n_views=2, beta_hist=None, same_as_current=False):
    from paper_2608_02134_gb300 import workloads
    wl = workloads.make("tiny")
    im = wl.image(0)
    f = lambda a: np.asarray(a, dtype=np.float64)
    hist = []
    for _ in range(n_views):
        if same_as_current:
            hist.append(dict(Q=f(im.queries), K=f(im.keys), V=f(im.values), W=f(wl.probe())))
        else:
            hist.append({k: f(a) for k, a in wl.history_view(0, len(hist)).items()})
    p = O.params() if beta_hist is None else O.params(beta_hist=beta_hist)
    args = (f(im.hidden), f(im.keys), f(im.values), f(im.queries), im.pos, f(wl.probe()),
            wl.gh, wl.gw, wl.K, p)
    return wl, O.compress(*args), O.compress(*args, history=hist), p


def test_view_patterns_combine_single_view_patterns():
    # blocks of the concatenated pattern are orthogonal, so
    # <u_h, u_g> = sum_v beta_v <U_h^v, U_g^v> with <U_h^v, U_g^v> = cos_v pre_v pre_v
    g = rng(11)
    H, T, N, r = 3, 2, 5, 4
    views = []
    for beta in (0.5, 0.2, 0.3):
        A = g.random((H, T, N))
        A /= A.sum(axis=2, keepdims=True)
        views.append((A, g.standard_normal((H, N, r)), g.random(H) + 0.1, beta))
    cos, pre, _ = O.view_patterns(views)
    dot = np.zeros((H, H))
    for A, Z, sigma, beta in views:
        c1, p1, _ = O.head_patterns(A, Z, sigma)
        dot += beta * c1 * np.outer(p1, p1)
    np.testing.assert_allclose(pre, np.sqrt(np.diag(dot)), rtol=1e-12)
    np.testing.assert_allclose(cos, dot / np.outer(pre, pre), rtol=1e-12)


def test_duplicate_views_keep_the_single_view_patterns():
    g = rng(12)
    H, T, N = 4, 3, 6
    A = g.random((H, T, N))
    Z = g.standard_normal((H, N, 4))
    sigma = g.random(H) + 0.1
    c1, p1, _ = O.head_patterns(A, Z, sigma)
    cos, pre, _ = O.view_patterns([(A, Z, sigma, 0.5), (A, Z, sigma, 0.25), (A, Z, sigma, 0.25)])
    np.testing.assert_allclose(cos, c1, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(pre, p1, rtol=1e-12)        # sqrt(0.5 + 0.25 + 0.25) = 1


def test_no_history_and_zero_history_mass_leave_the_step_unchanged():
    wl, base, empty, _ = _tiny_with_history(n_views=0)
    np.testing.assert_array_equal(empty.support, base.support)
    np.testing.assert_allclose(empty.heads.omega, base.heads.omega, rtol=1e-12)
    np.testing.assert_allclose(empty.clients.C, base.clients.C, rtol=1e-12, atol=1e-18)
    wl, base, zero, _ = _tiny_with_history(n_views=2, beta_hist=0.0)
    np.testing.assert_array_equal(zero.support, base.support)
    np.testing.assert_allclose(zero.heads.omega, base.heads.omega, rtol=1e-12)
    assert not zero.clients.C[zero.clients.views[1]].any()


def test_history_views_add_client_blocks_with_their_masses():
    wl, base, res, p = _tiny_with_history(n_views=2)
    H, T = wl.H, int(wl.T[0])
    cm = res.clients
    assert cm.C.shape[0] == 3 * H * T + wl.N + p["landmarks"] ** 2
    masses = [p["beta_G"], p["beta_hist"] / 2, p["beta_hist"] / 2]
    for v, beta in enumerate(masses):
        blk = cm.C[cm.views[v]]
        assert blk.shape == (H * T, wl.N)
        act = [res.activeG] + [hv[5] for hv in res.history]
        want = beta * np.outer(res.heads.omega, res.nu) * act[v]
        np.testing.assert_allclose(blk.sum(axis=1), want.reshape(-1), rtol=1e-12, atol=1e-18)
    # the message energy stays the current view's (Eq. (cond-grounded-energy))
    e, _ = O.message_energy(res.unorm, res.heads.omega, res.nu)
    np.testing.assert_allclose(res.e, e, rtol=1e-14)
    S = res.support
    assert S.size == wl.K and np.all(np.diff(S) > 0)


def test_duplicated_current_view_as_history_keeps_head_weights():
    wl, base, res, _ = _tiny_with_history(n_views=2, same_as_current=True)
    np.testing.assert_array_equal(res.heads.centres, base.heads.centres)
    np.testing.assert_allclose(res.heads.omega, base.heads.omega, rtol=1e-12)


# --------------------------------------------------------------------------
# Cached path: dense prefix layers at the kept rows (appendix "Index map and
# physical token accounting")
# --------------------------------------------------------------------------
def test_prefix_kv_gather_is_the_index_map_layer_by_layer():
    from paper_2608_02134_gb300 import workloads
    wl = workloads.make("tiny", K=20, T=6)
    im = wl.image(0)
    f = lambda a: np.asarray(a, dtype=np.float64)
    prefix = [(f(wl.prefix_kv(0, l)["K"]), f(wl.prefix_kv(0, l)["V"])) for l in range(3)]
    res = O.compress(f(im.hidden), f(im.keys), f(im.values), f(im.queries), im.pos,
                     f(wl.probe()), wl.gh, wl.gw, wl.K, prefix=prefix)
    N, T = wl.N, 6
    kept = list(res.support) + list(range(N, N + T))          # brute force, row by row
    assert res.out_prefix_kv.shape == (3, 2, wl.K + T, wl.Hkv, wl.d)
    for l, (Kl, Vl) in enumerate(prefix):
        for r, src in enumerate(kept):
            assert np.array_equal(res.out_prefix_kv[l, 0, r], Kl[src])
            assert np.array_equal(res.out_prefix_kv[l, 1, r], Vl[src])
    # the boundary layer's own K/V follow the same map
    assert np.array_equal(res.out_kv[0], f(im.keys)[kept])
    # identity budget: every prefix layer unchanged
    idn = O.compress(f(im.hidden), f(im.keys), f(im.values), f(im.queries), im.pos,
                     f(wl.probe()), wl.gh, wl.gw, wl.N, prefix=prefix)
    for l, (Kl, Vl) in enumerate(prefix):
        assert np.array_equal(idn.out_prefix_kv[l, 0], Kl) and np.array_equal(idn.out_prefix_kv[l, 1], Vl)
    none = O.compress(f(im.hidden), f(im.keys), f(im.values), f(im.queries), im.pos,
                      f(wl.probe()), wl.gh, wl.gw, wl.K)
    assert none.out_prefix_kv.shape[0] == 0


# --------------------------------------------------------------------------
# Multi-image prompts (Sec. 3.1 budget, Sec. 3.3 seeding, appendix Eq.
# (cond-aux-clients) with 1[I_i = I_m], same-image assignment)
# --------------------------------------------------------------------------
def _multi_case(I=3, gh=4, gw=5, D=6, seed=80):
    r = rng(seed)
    N = I * gh * gw
    h = r.standard_normal((N, D))
    return h, N


def test_multi_image_appearance_rows_stay_in_their_image():
    I, gh, gw = 3, 4, 5
    h, N = _multi_case(I, gh, gw)
    cos = O.cosine_matrix(h, P)
    PV = O.appearance_clients(cos, P, n_images=I)
    Ng = gh * gw
    for k in range(I):
        blk = slice(k * Ng, (k + 1) * Ng)
        # each image's block is the single-image bank of that image alone
        np.testing.assert_allclose(PV[blk, blk], O.appearance_clients(cos[blk, blk], P), rtol=1e-13)
        off = np.ones(N, bool)
        off[blk] = False
        assert np.all(PV[blk][:, off] == 0.0)
    np.testing.assert_allclose(PV.sum(axis=1), 1.0, rtol=1e-13)


def test_multi_image_spatial_landmarks_per_image():
    I, gh, gw = 2, 6, 6
    PS = O.spatial_clients(gh, gw, P, n_images=I)
    one = O.spatial_clients(gh, gw, P)
    L2, Ng = one.shape
    assert PS.shape == (I * L2, I * Ng)
    for k in range(I):
        for k2 in range(I):
            blk = PS[k * L2:(k + 1) * L2, k2 * Ng:(k2 + 1) * Ng]
            if k == k2:
                np.testing.assert_array_equal(blk, one)
            else:
                assert np.all(blk == 0.0)
    # bank mass: beta_S shared by all I * L^2 rows
    hvis = rng(81).standard_normal((I * Ng, 5))
    cm = O.client_matrix(np.zeros((1, 1, I * Ng)), np.zeros((1, 1), bool), np.ones(1), np.ones(1),
                         O.appearance_clients(O.cosine_matrix(hvis, P), P, I), PS, P)
    assert cm.C[cm.banks["spatial"]].sum() == pytest.approx(P["beta_S"], rel=1e-13)


def test_multi_image_seeds_are_each_images_best_singleton():
    I, Ng, M = 3, 12, 40
    C = _rand_C(M, I * Ng, 82)
    u = C.sum(axis=0)
    sel = O.select_support(C, 10, P, n_images=I)
    seed = sel.rounds[0]
    assert seed.seed and list(seed.batch) == sel.order[:I]
    for k in range(I):   # brute force: largest column sum of image k, lowest index on ties
        best = max(range(k * Ng, (k + 1) * Ng), key=lambda i: (u[i], -i))
        assert sel.order[k] == best
    assert len(sel.order) == 10 and len(set(sel.order)) == 10
    # a budget below the image count: one carrier per image, the seeds
    assert O.budget(2, I * Ng, I) == I
    sel2 = O.select_support(C, O.budget(2, I * Ng, I), P, n_images=I)
    assert sel2.order == sel.order[:I]
    # a single image: no seed round, the plain solver
    s1 = O.select_support(C, 10, P)
    assert not s1.rounds[0].seed


def test_multi_image_assignment_is_same_image():
    I, gh, gw = 3, 4, 5
    h, N = _multi_case(I, gh, gw, seed=83)
    Ng = gh * gw
    cos = O.cosine_matrix(h, P)
    S = np.array([1, 7, 22, 33, 41, 55])   # image 0: 1, 7; image 1: 22, 33; image 2: 41, 55
    a = O.assign_population(cos, S, gh, gw, P, n_images=I)
    img = np.arange(N) // Ng
    assert np.all(img[a.pi] == img)          # clusters never cross images
    assert np.all(a.pi[S] == S)
    for i in range(N):                        # the gap over same-image carriers only
        if i in S:
            continue
        Si = S[img[S] == img[i]]
        v = sorted(cos[i, Si], reverse=True)
        assert a.delta[i] == pytest.approx(v[0] - v[1], abs=1e-15)
    # a plain nearest neighbour when the gate is closed, within the image
    b = O.assign_population(cos, S, gh, gw, O.params(gate_scale=1e9), n_images=I)
    for i in range(N):
        if i not in S:
            Si = S[img[S] == img[i]]
            assert b.pi[i] == Si[int(np.argmax(cos[i, Si]))]


def test_multi_image_compress_invariants():
    from paper_2608_02134_gb300 import workloads
    wl = workloads.make("tiny", I=2, gh=6, gw=6, T=5, K=9)
    im = wl.image(0)
    f = lambda a: np.asarray(a, dtype=np.float64)
    res = O.compress(f(im.hidden), f(im.keys), f(im.values), f(im.queries), im.pos,
                     f(wl.probe()), wl.gh, wl.gw, wl.K, n_images=2)
    N, Ng = wl.N, wl.Ng
    img = np.arange(N) // Ng
    assert res.K == 9 and res.support.size == 9
    assert set(img[res.support]) == {0, 1}
    assert np.all(img[res.assignment.pi] == img)
    # transport conserves each image's population mass
    for k in range(2):
        Sk = res.support[img[res.support] == k]
        slot = np.searchsorted(res.support, Sk)
        assert res.transport.mass[slot].sum() == pytest.approx(res.m[img == k].sum(), rel=1e-12)
    # one image is the single-image path
    wl1 = workloads.make("tiny")
    im1 = wl1.image(0)
    r1 = O.compress(f(im1.hidden), f(im1.keys), f(im1.values), f(im1.queries), im1.pos,
                    f(wl1.probe()), wl1.gh, wl1.gw, wl1.K, n_images=1)
    r0 = O.compress(f(im1.hidden), f(im1.keys), f(im1.values), f(im1.queries), im1.pos,
                    f(wl1.probe()), wl1.gh, wl1.gw, wl1.K)
    assert np.array_equal(r1.support, r0.support) and np.array_equal(r1.out_hidden, r0.out_hidden)


def test_multi_image_assignment_uses_each_images_own_grid():
    """Two copies of one image with mirrored supports assign exactly like the
    single image: same gaps, gate and kappa (coordinates are per image grid)."""
    gh, gw, Ng = 4, 5, 20
    h0 = rng(84).standard_normal((Ng, 3))
    S0 = np.array([2, 9, 13, 18])
    single = O.assign_population(O.cosine_matrix(h0, P), S0, gh, gw, P)
    assert single.s_x > 0.5 and np.max(single.g[np.setdiff1d(np.arange(Ng), S0)]) > 0.1
    h = np.concatenate([h0, h0])
    both = O.assign_population(O.cosine_matrix(h, P), np.concatenate([S0, S0 + Ng]), gh, gw, P,
                               n_images=2)
    assert both.s_x == pytest.approx(single.s_x, rel=1e-13)
    for k in range(2):
        blk = slice(k * Ng, (k + 1) * Ng)
        np.testing.assert_array_equal(both.pi[blk], single.pi + k * Ng)
        np.testing.assert_allclose(both.kappa_best[blk], single.kappa_best, rtol=1e-13)


# --------------------------------------------------------------------------
# Long prefixes: the bounded appearance bank (appendix "Appearance and
# spatial clients", last paragraph; Table "Shared GMC configuration",
# long-prefix row)
# --------------------------------------------------------------------------
def _orthogonal_pm1(n: int, seed: int) -> np.ndarray:
    """A +-1 matrix with R R^T = R^T R = n I that is not symmetric: a
    Sylvester-Hadamard matrix with permuted, sign-flipped columns."""
    from scipy.linalg import hadamard
    r = rng(seed)
    return (hadamard(n)[:, r.permutation(n)] * r.choice([-1.0, 1.0], size=n)[None, :]).astype(float)


def test_bounded_client_tokens_are_uniformly_spaced():
    np.testing.assert_array_equal(O.bounded_client_tokens(1296, 4096), np.arange(1296))
    for N, M in [(15876, 4096), (1600, 512), (4097, 4096), (10, 3)]:
        c = O.bounded_client_tokens(N, M)
        assert c.size == M and c[0] == 0 and c[-1] < N
        gaps = np.diff(c)
        assert set(gaps.tolist()) <= {N // M, -(-N // M)}
        assert len(set(c.tolist())) == M


def test_projected_cosines_equal_exact_under_an_orthogonal_map():
    """R R^T = n I preserves inner products up to the factor n, which the
    normalisation removes: projected cosines are the exact cosines."""
    D = 64
    R = _orthogonal_pm1(D, 3)
    assert not np.array_equal(R, R.T)
    h = rng(4).standard_normal((30, D)) * rng(5).uniform(0.1, 10, size=(30, 1))
    xt = O.projected_states(h, R, P)
    np.testing.assert_allclose(xt @ xt.T, O.cosine_matrix(h, P), atol=1e-13)
    np.testing.assert_allclose(np.linalg.norm(xt, axis=1), 1.0, rtol=1e-14)


def test_projected_states_ignore_the_maps_null_space_and_scale():
    r, D = 8, 40
    R = rng(6).choice([-1.0, 1.0], size=(r, D))
    h = rng(7).standard_normal((12, D))
    # a component in the null space of R (orthogonal to every row of R)
    q, _ = np.linalg.qr(R.T)                       # [D, r]: the row space of R
    v = rng(8).standard_normal((12, D))
    v -= (v @ q) @ q.T
    np.testing.assert_allclose(O.projected_states(h + 5 * v, R, P), O.projected_states(h, R, P),
                               atol=1e-12)
    np.testing.assert_allclose(O.projected_states(h, R / math.sqrt(r), P),
                               O.projected_states(h, R, P), atol=1e-14)


def test_random_rademacher_cosines_obey_a_johnson_lindenstrauss_bound():
    """Rank 128 keeps cosines of random states within a few 1/sqrt(128)."""
    D, r = 512, 128
    R = rng(9).choice([-1.0, 1.0], size=(r, D))
    h = rng(10).standard_normal((40, D))
    h[20:] = h[:20] + 0.5 * rng(11).standard_normal((20, D))  # correlated pairs too
    err = np.abs(O.projected_states(h, R, P) @ O.projected_states(h, R, P).T - O.cosine_matrix(h, P))
    assert err.max() < 0.45 and err.mean() < 0.12


def test_bounded_rows_are_the_exact_rows_of_their_client_tokens():
    """Under an orthogonal map every bounded appearance row is the exact
    bank's row of its client token, for one image and per image."""
    D, N = 32, 60
    R = _orthogonal_pm1(D, 12)
    h = rng(13).standard_normal((N, D))
    for n_img in (1, 2):
        exact = O.appearance_clients(O.cosine_matrix(h, P), P, n_img)
        c = O.bounded_client_tokens(N, 17)
        bounded = O.bounded_appearance_clients(O.projected_states(h, R, P), c, P, n_img)
        assert bounded.shape == (17, N)
        np.testing.assert_allclose(bounded, exact[c], rtol=1e-11, atol=1e-300)


def test_bounded_bank_rows_carry_beta_v_over_m_v():
    H, T, N, MV = 2, 3, 20, 7
    PG = rng(14).uniform(size=(H, T, N))
    PG /= PG.sum(axis=2, keepdims=True)
    PV = rng(15).uniform(size=(MV, N))
    PV /= PV.sum(axis=1, keepdims=True)
    PS = O.spatial_clients(4, 5, P)
    cm = O.client_matrix(PG, np.ones((H, T), bool), np.full(H, 0.5), np.full(T, 1 / 3), PV, PS, P)
    assert cm.C.shape == (H * T + MV + PS.shape[0], N)
    rows = cm.C[cm.banks["appearance"]].sum(axis=1)
    np.testing.assert_allclose(rows, P["beta_V"] / MV, rtol=1e-14)
    assert cm.C[cm.banks["spatial"]].sum() == pytest.approx(P["beta_S"], rel=1e-13)


def test_support_column_cosines_give_the_full_matrix_assignment():
    gh, gw = 5, 6
    h = rng(16).standard_normal((gh * gw, 7))
    S = np.array([1, 4, 11, 17, 22, 29])
    full = O.assign_population(O.cosine_matrix(h, P), S, gh, gw, P)
    cols = O.support_cosines(h, S, P)
    np.testing.assert_allclose(cols, O.cosine_matrix(h, P)[:, S], atol=1e-15)
    part = O.assign_population(cols, S, gh, gw, P, support_cols=True)
    np.testing.assert_array_equal(part.pi, full.pi)
    np.testing.assert_allclose(part.delta, full.delta, atol=1e-15)
    assert part.s_x == full.s_x


def test_long_prefix_step_equals_the_exact_step_under_an_orthogonal_map():
    """With an orthogonal +-1 map of rank D and every token a client, the
    bounded-bank step is the exact-bank step (same support, assignment and
    outputs); with fewer clients it keeps its invariants."""
    from paper_2608_02134_gb300 import workloads
    wl = workloads.make("tiny")
    im = wl.image(0)
    f = lambda a: np.asarray(a, dtype=np.float64)  # noqa: E731
    args = (f(im.hidden), f(im.keys), f(im.values), f(im.queries), im.pos, f(wl.probe()),
            wl.gh, wl.gw, wl.K)
    R = _orthogonal_pm1(wl.D, 17)
    exact = O.compress(*args)
    bounded = O.compress(*args, long_prefix=dict(R=R, max_clients=wl.N))
    np.testing.assert_array_equal(bounded.support, exact.support)
    np.testing.assert_array_equal(bounded.assignment.pi, exact.assignment.pi)
    np.testing.assert_allclose(bounded.out_hidden, exact.out_hidden, rtol=1e-12, atol=1e-12)
    few = O.compress(*args, long_prefix=dict(R=R, max_clients=16))
    assert few.clients.banks["appearance"].stop - few.clients.banks["appearance"].start == 16
    assert few.support.size == wl.K and np.all(np.diff(few.support) > 0)
    assert few.transport.mass.sum() == pytest.approx(few.m.sum(), rel=1e-12)
    assert np.all(np.isin(few.assignment.pi, few.support))
