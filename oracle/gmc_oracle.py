"""Plain fp64 CPU oracle of the GMC layer-boundary compression step.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
module.  The CUDA library never calls it, and it imports nothing from the
CUDA package: the two paths share no code.  It is deliberately slow and
literal: every function follows one step of the paper (Grounded Message
Coreset Pruning, arXiv 2608.02134) in the paper's order and notation, in
float64, with numpy primitives (matmul, exp, sort) as the only library steps.

Paper passages followed (section / equation labels of the paper):
  * Sec. 3.1 budget rule ``K = min{N, max{K_r, I}}``.
  * Sec. 3.2, Eq. (1) mass coordinate, Eq. (2) grounded clients; Appendix
    "Native message clients": Eq. (cond-native-message), (cond-mass-coordinate),
    (cond-grounded-client), (cond-head-pattern), (cond-head-weight).
  * Appendix "Appearance and spatial clients": Eq. (cond-aux-clients),
    (cond-coverage), (cond-effective-bank-mass).
  * Sec. 3.3 Eq. (3) facility location, Eq. (4) responsibility; Appendix
    "Batched complementary support": Eq. (cond-responsibility) and the
    totality rule.
  * Sec. 3.4 Eq. (5); Appendix "Population assignment and transport":
    Eq. (cond-assignment), (cond-transport), (cond-grounded-energy),
    (cond-population-gate).
  * Algorithm 1 (steps 2-6) and Appendix "Index map and physical token
    accounting" for the compaction.
  * Table "Shared GMC configuration" for every constant.
  * Sec. 4.1 Eq. (6) and Appendix Eq. (cond-batched-bound),
    (cond-final-cert), (cond-bank-mixture) for the diagnostics.

Readings taken where the paper is silent or ambiguous:
  * The probe enters as ``W_h = O_h P`` (d x 4); only ||Z_h[i]|| and
    ||Z_h||_F are used.
  * Softmax keys: all N visual keys plus text keys 0..t (causal), scale
    1/sqrt(d).  Sequence layout is ``[N visual][T text]``.
  * Grounded client row (h, t) carries weight beta_G * omega_h * nu_t.
  * Head patterns use atoms over all (t, i), unweighted by nu; clustering
    ties go to the lowest head index, head-to-centre ties to the earliest
    centre.
  * Appearance state x_i = h_i / max(||h_i||, 1e-12) of the raw boundary state.
  * Grid coordinates ((r+0.5)/gh, (c+0.5)/gw); landmarks ((a+0.5)/16, (b+0.5)/16).
  * Pool = top-min(4b, #{u_i > 0}) unselected tokens by gain; batch =
    top-min(b, |pool|, K-|S|) by responsibility score; ties to the lowest
    token index; an empty pool fills the rest in ascending index order.
  * Local ambiguity g_i = exp(-(delta_i / 0.05)^8); delta_i = 0 when the
    support has one element.
  * Transport blend tau_j = 1 (appendix form); rms(u) = sqrt(mean u^2),
    epsilon 1e-6.
  * Multi-image prompts: I images of equal grids lie one after another in
    the visual segment; coordinates, landmarks and the assignment's spatial
    term use each image's own grid; the seed round picks one max-gain token
    per image before the responsibility rounds.
  * Historical message views (optional): the configuration table's
    "current/history mass 0.5/0.5" is read as a current-view grounded mass
    beta_G = 0.5 and a history mass beta_hist = 0.5 shared equally by the
    completed views; each view carries its own layer's queries, keys, values
    and probe W = O_h P; omega_h and nu_t weight every view's rows; the
    message energy is the current view's only.
  * Long prefixes (bounded appearance bank): the rank-r Rademacher map R
    [r, D] (+-1 entries, numpy default_rng(104729), an input like the probe)
    acts on the raw boundary state and the result is normalised,
    x~_i = R h_i / ||R h_i||; the M_V = min(N, 4096) clients are the tokens
    floor(m N / M_V); their rows carry beta_V / M_V; the assignment uses the
    cosines of the unprojected states against the support only.

Pins (tests/test_oracle_pins.py; the paper prints no worked numeric example,
so every function is pinned by a closed form, an invariant, a bound of the
paper, a hand-worked case or brute force on tiny inputs, never by itself):
  * budget: the totality rule on every (K_r, N) corner.
  * message_slice: explicit per-element loops; causal keys and the native
    (not renormalised) visual mass; one query is a plain softmax.
  * orthonormal_probe / probe_values: orthonormal columns; rotation
    invariance of ||Z||; the sigma floor closed form (V = 0 => P^G prop. to A).
  * atom_norms / grounded_clients: a hand example; a zero-energy row is
    inactive.
  * query_weights: the terminal query counts double, weights sum to one.
  * head_patterns / head_clusters: identical heads form one cluster with
    uniform weights; orthogonal families get equal cluster mass; a
    hand-worked farthest-first case; weights follow 1 / (dispersion + eps).
  * message_energy: closed form and the uniform fallback.
  * cosine_matrix / appearance_clients: the Gibbs modal ratio.
  * grid_coords / landmark_coords / spatial_clients: normalised cell centres,
    landmark-grid ratios.
  * client_matrix / bank_saturation: bank masses and effective shares, row
    masses from head and query weights.
  * facility_value: Eq. (7) coverage-to-quantization bound; monotone and
    submodular by brute force.
  * select_support / stable_top / batched_certificate: Eq. (6) certificate and
    the greedy (1 - 1/e) bound against brute-force optima; exact cardinality;
    the zero-gain fill; a hand-worked responsibility round
    (tests/golden/responsibility_round.txt); trivial supports.
  * assign_population: cosine nearest neighbour when s_x = 0; the gap-gate
    closed form and Eq. (cond-assignment-bound); one representative; a
    hand-worked case at s_x = 1 - 1/e where the spatial term, its ambiguity
    gate and the grid coordinates each decide one representative
    (tests/golden/assignment_spatial_gate.txt).
  * population_weights / transport / rms: positivity, mass and first-moment
    conservation (Eq. (cond-population-moment)), centroid optimality
    (Eq. (cond-centroid-optimum)), RMS restoration and its bound; energies,
    weights and a two-cluster transport worked by hand at s_x = 1 - 1/e
    (tests/golden/population_transport.txt).
  * compaction_rows / compress: K = N identity; end-to-end invariants on the
    tiny configuration.
  * multi-image prompts (image_index and the n_images arguments): each
    image's appearance block is the single-image bank of that image and zero
    elsewhere; spatial landmarks repeat per image, block-diagonal; the seeds
    are every image's best singleton gain (brute force) and a budget below
    the image count keeps exactly them; clusters never cross images and the
    gap uses same-image carriers only (brute force); two copies of one image
    assign exactly like the image alone; one image is the single-image path.
  * gather_prefix_kv: the gathered prefix rows are the source rows at the
    compaction index map, bit for bit, layer by layer (brute force), and the
    identity budget returns every layer unchanged.
  * view_patterns / client_matrix_views / compress(history=...): the
    multi-view pattern Gram equals the beta-weighted sum of single-view
    pattern Grams; duplicated views keep the single-view cosines and head
    weights; no history or zero history mass leaves the step unchanged; each
    view's rows carry its mass; the energy stays the current view's.
  * bounded_client_tokens / projected_states / bounded_appearance_clients /
    support_cosines / compress(long_prefix=...): uniform spacing (count,
    first token, gaps of floor or ceil N/M_V); under an orthogonal +-1 map
    (a signed, column-permuted Sylvester-Hadamard matrix, D = r) projected
    cosines equal the exact ones, so every bounded row is the exact bank's
    row of its client token and, with M_V >= N, the whole step equals the
    exact-bank step; a null-space component of R leaves x~ unchanged; a
    Johnson-Lindenstrauss bound on random maps; support-column cosines give
    the full-matrix assignment; appearance rows carry beta_V / M_V each.

Discrete choices (pool, batch, head centres, assignment) are recorded together
with the fp64 values that decide them.  Every choice can also be *forced*
(``forced=`` arguments): the oracle then continues from the given choice
instead of its own, so a test can check a choice made elsewhere against these
values and keep comparing after a near-tie without the tie cascading.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

# Table "Shared GMC configuration" (fixed-token settings) plus the readings
# listed in the module docstring.
DEFAULTS = dict(
    probe_rank=4,            # rank-4 probe
    lambda_mass=1.0,         # lambda_mass = 1
    eps_mass=1e-8,           # epsilon_mass = 1e-8
    beta_G=0.5,              # current-view grounded mass
    beta_hist=0.5,           # historical-view grounded mass, split equally over the views
    beta_V=0.5,              # appearance mass
    beta_S=0.25,             # spatial mass
    tau_v=0.2,               # appearance temperature
    tau_s=0.02,              # spatial temperature
    landmarks=16,            # 16 x 16 landmarks
    max_head_clusters=4,     # at most four head clusters
    head_eps=0.05,           # (d_h + 0.05)^-1 in Eq. (cond-head-weight)
    terminal_q_weight=2.0,   # terminal prompt query counts twice
    batch_b=16,              # responsibility batch b
    pool_mult=4,             # candidate pool 4b
    resp_temp=0.1,           # responsibility temperature
    resp_eps=1e-12,          # epsilon of Eq. (4)
    assign_spatial_w=0.5,    # spatial weight 0.5
    gate_scale=0.08,         # gate (0.08, 8)
    gate_pow=8.0,
    ambig_margin=0.05,       # ambiguity margin 0.05
    pop_strength=0.5,        # grounded population strength alpha
    rms_eps=1e-6,            # epsilon of R_j
    norm_eps=1e-12,          # epsilon of h / max(||h||, eps)
)


def params(**overrides) -> dict:
    p = dict(DEFAULTS)
    for k, v in overrides.items():
        if k not in p:
            raise KeyError(f"unknown GMC parameter {k!r}")
        p[k] = v
    return p


# ---------------------------------------------------------------------------
# a1: budget (Sec. 3.1; Appendix "Batched complementary support", totality rule)
# ---------------------------------------------------------------------------
def budget(K_r: int, N: int, n_images: int = 1) -> int:
    """K = min{N, max{K_r, I}}."""
    return int(min(N, max(int(K_r), int(n_images))))


# ---------------------------------------------------------------------------
# a2: native boundary attention slice (Eq. (cond-native-message))
# ---------------------------------------------------------------------------
def kv_head_of(h: int, H: int, Hkv: int) -> int:
    """Grouped-query attention: query head h reads key/value head h // (H/Hkv)."""
    return h // (H // Hkv)


def message_slice(Q: np.ndarray, Kall: np.ndarray, N: int) -> np.ndarray:
    """A_h = softmax((Q_h K_h^T + M_causal)/sqrt(d_h))[:, visual columns].

    Q: [T, H, d] text queries; Kall: [N+T, Hkv, d] keys (visual rows first).
    Text query t sits at sequence position N+t and sees every visual key and
    text keys 0..t.  The softmax is the native one over all of those keys;
    only its visual columns are kept, without renormalising them.
    Returns A: [H, T, N].
    """
    T, H, d = Q.shape
    L, Hkv, _ = Kall.shape
    assert L == N + T
    allowed = np.zeros((T, L), dtype=bool)
    allowed[:, :N] = True
    for t in range(T):
        allowed[t, N:N + t + 1] = True
    A = np.empty((H, T, N))
    for h in range(H):
        g = kv_head_of(h, H, Hkv)
        S = (Q[:, h, :] @ Kall[:, g, :].T) / math.sqrt(d)
        S = np.where(allowed, S, -np.inf)
        S = S - S.max(axis=1, keepdims=True)
        P = np.exp(S)
        P /= P.sum(axis=1, keepdims=True)
        A[h] = P[:, :N]
    return A


# ---------------------------------------------------------------------------
# a3: probe values and the mass coordinate (Eq. (1), Eq. (cond-mass-coordinate))
# ---------------------------------------------------------------------------
def orthonormal_probe(G: np.ndarray) -> np.ndarray:
    """P from the reduced QR factorisation G = P R of a Gaussian draw G."""
    P, _ = np.linalg.qr(G, mode="reduced")
    return P


def probe_values(Vvis: np.ndarray, W: np.ndarray, H: int, p: dict):
    """Z_h = (V_h O_h) P = V_h W_h and sigma_h.

    Vvis: [N, Hkv, d] visual values; W: [H, d, r] with W_h = O_h P.
    sigma_h = sqrt(lambda_mass) * max{||Z_h||_F / sqrt(N r), eps_mass}.
    Returns Z [H, N, r], sigma [H].
    """
    N, Hkv, d = Vvis.shape
    r = W.shape[2]
    Z = np.empty((H, N, r))
    sigma = np.empty(H)
    for h in range(H):
        Z[h] = Vvis[:, kv_head_of(h, H, Hkv), :] @ W[h]
        fro = math.sqrt(float(np.sum(Z[h] * Z[h])))
        sigma[h] = math.sqrt(p["lambda_mass"]) * max(fro / math.sqrt(N * r), p["eps_mass"])
    return Z, sigma


# ---------------------------------------------------------------------------
# a4: grounded atoms and clients (Eq. (2), Eq. (cond-grounded-client))
# ---------------------------------------------------------------------------
def atom_norms(A: np.ndarray, Z: np.ndarray, sigma: np.ndarray) -> np.ndarray:
    """||u_i^{h,t}|| with u_i^{h,t} = A_h[t,i] [Z_h[i]; sigma_h].  Returns [H, T, N]."""
    g = np.sqrt(np.sum(Z * Z, axis=2) + sigma[:, None] ** 2)   # [H, N]
    return A * g[:, None, :]


def grounded_clients(unorm: np.ndarray):
    """P^G_{h,t}(i) = ||u_i|| / sum_j ||u_j|| for active rows; zero rows stay inactive.

    Returns PG [H, T, N] and the active indicator a [H, T].
    """
    tot = unorm.sum(axis=2)
    active = tot > 0
    PG = np.zeros_like(unorm)
    PG[active] = unorm[active] / tot[active][:, None]
    return PG, active


# ---------------------------------------------------------------------------
# a5: query weights, head clusters, head weights, message energy
# ---------------------------------------------------------------------------
def query_weights(T: int, p: dict) -> np.ndarray:
    """nu_t: the terminal prompt query counts terminal_q_weight times, then normalise."""
    w = np.ones(T)
    w[T - 1] = p["terminal_q_weight"]
    return w / w.sum()


def head_patterns(A: np.ndarray, Z: np.ndarray, sigma: np.ndarray):
    """Eq. (cond-head-pattern) for the current view.

    U_h collects the atoms u_i^{h,t} in R^{r+1} over all (t, i), divided by
    their mean norm; the pattern is U_h / ||U_h||.  Returns the pattern cosine
    matrix [H, H] and the pre-normalisation norms ||U_h|| [H].  A head whose
    atoms are all zero has the zero pattern (norm 0, cosine 0).
    """
    H, T, N = A.shape
    vecs = []
    for h in range(H):
        zs = np.concatenate([Z[h], np.full((N, 1), sigma[h])], axis=1)     # [N, r+1]
        atoms = A[h][:, :, None] * zs[None, :, :]                          # [T, N, r+1]
        mean_norm = float(np.mean(np.sqrt(np.sum(atoms * atoms, axis=2))))
        vecs.append(atoms.reshape(-1) / mean_norm if mean_norm > 0 else np.zeros(atoms.size))
    U = np.stack(vecs)
    pre = np.sqrt(np.sum(U * U, axis=1))
    unit = np.zeros_like(U)
    nz = pre > 0
    unit[nz] = U[nz] / pre[nz][:, None]
    return unit @ unit.T, pre, unit


def view_patterns(views):
    """Eq. (cond-head-pattern) over message views.

    ``views`` lists (A, Z, sigma, beta) per view (current first).  U_h^v
    collects the atoms of head h in view v divided by their mean norm (the
    zero vector when every atom is zero); the pattern is
    concat_v [sqrt(beta_v) vec(U_h^v)] divided by its norm.  Returns the
    pattern cosine matrix [H, H], the pre-normalisation norms [H] and the unit
    patterns.
    """
    H = views[0][0].shape[0]
    rows = [[] for _ in range(H)]
    for A, Z, sigma, beta in views:
        _, T, N = A.shape
        for h in range(H):
            zs = np.concatenate([Z[h], np.full((N, 1), sigma[h])], axis=1)     # [N, r+1]
            atoms = A[h][:, :, None] * zs[None, :, :]                          # [T, N, r+1]
            mean_norm = float(np.mean(np.sqrt(np.sum(atoms * atoms, axis=2))))
            Uv = atoms.reshape(-1) / mean_norm if mean_norm > 0 else np.zeros(atoms.size)
            rows[h].append(math.sqrt(beta) * Uv)
    U = np.stack([np.concatenate(r) for r in rows])
    pre = np.sqrt(np.sum(U * U, axis=1))
    unit = np.zeros_like(U)
    nz = pre > 0
    unit[nz] = U[nz] / pre[nz][:, None]
    return unit @ unit.T, pre, unit


@dataclass
class HeadClusters:
    centres: list           # centre heads in the order farthest-first chose them
    assign: np.ndarray      # [H] index into ``centres`` of each head's cluster
    omega: np.ndarray       # [H] head weights
    cos: np.ndarray         # [H, H] pattern cosines used for every choice
    pre_norm: np.ndarray    # [H] pre-normalisation pattern norms
    dispersion: np.ndarray  # [H] d_h = 1 - u_h^T mu_c(h)
    n_clusters: int


def head_clusters(A, Z, sigma, p, forced_centres=None, forced_assign=None,
                  views=None) -> HeadClusters:
    """Farthest-first cosine clustering and Eq. (cond-head-weight).

    First centre: the largest pre-normalisation pattern.  Then, until
    min(max_head_clusters, H) centres exist, add the head whose maximum cosine
    to the existing centres is smallest.  Each head joins its most similar
    centre.  omega_h = (1/C) (d_h + eps)^-1 / sum_{g in c(h)} (d_g + eps)^-1
    with C the number of nonempty clusters and d_h = 1 - u_h^T mu_c, mu_c the
    normalised mean pattern of the cluster.  With ``views`` (see
    view_patterns) the patterns span every message view.
    """
    cos, pre, unit = head_patterns(A, Z, sigma) if views is None else view_patterns(views)
    H = cos.shape[0]
    n_c = min(p["max_head_clusters"], H)
    if forced_centres is not None:
        centres = [int(c) for c in forced_centres]
    else:
        centres = [int(np.lexsort((np.arange(H), -pre))[0])]
        while len(centres) < n_c:
            rest = [h for h in range(H) if h not in centres]
            mc = np.array([max(cos[h, c] for c in centres) for h in rest])
            order = np.lexsort((np.array(rest), mc))
            centres.append(rest[int(order[0])])
    if forced_assign is not None:
        assign = np.asarray(forced_assign, dtype=np.int64)
    else:
        sims = cos[:, centres]                                   # [H, n_c]
        assign = np.array([int(np.lexsort((np.arange(len(centres)), -sims[h]))[0])
                           for h in range(H)])
    members = [np.flatnonzero(assign == k) for k in range(len(centres))]
    C = sum(1 for m in members if m.size > 0)
    omega = np.zeros(H)
    disp = np.zeros(H)
    for m in members:
        if m.size == 0:
            continue
        mu = unit[m].sum(axis=0)
        mu_n = float(np.linalg.norm(mu))
        mu = mu / mu_n if mu_n > 0 else mu
        d = 1.0 - unit[m] @ mu
        disp[m] = d
        inv = 1.0 / (d + p["head_eps"])
        omega[m] = (1.0 / C) * inv / inv.sum()
    return HeadClusters(centres, assign, omega, cos, pre, disp, C)


def message_energy(unorm: np.ndarray, omega: np.ndarray, nu: np.ndarray):
    """Eq. (cond-grounded-energy) with r_i^{h,t} = sqrt(nu_t) u_i^{h,t}.

    e_i = (sum_h omega_h sum_t nu_t ||u_i^{h,t}||^2)^{1/2};
    ebar_i = e_i / mean_j e_j, or 1 for every i when that mean is zero.
    """
    e2 = np.einsum("h,t,hti->i", omega, nu, unorm * unorm)
    e = np.sqrt(e2)
    mean = float(e.mean())
    ebar = e / mean if mean > 0 else np.ones_like(e)
    return e, ebar


# ---------------------------------------------------------------------------
# a6/a7: appearance and spatial clients (Eq. (cond-aux-clients))
# ---------------------------------------------------------------------------
def unit_states(hvis: np.ndarray, p: dict) -> np.ndarray:
    """x_i = h_i / max(||h_i||, eps)."""
    n = np.sqrt(np.sum(hvis * hvis, axis=1))
    return hvis / np.maximum(n, p["norm_eps"])[:, None]


def cosine_matrix(hvis: np.ndarray, p: dict) -> np.ndarray:
    x = unit_states(hvis, p)
    return x @ x.T


def image_index(N: int, n_images: int = 1) -> np.ndarray:
    """Image I_i of every visual token: n_images equal grids laid out one after
    another (tokens [k N/I, (k+1) N/I) belong to image k)."""
    return np.arange(N) // (N // n_images)


def appearance_clients(cos: np.ndarray, p: dict, n_images: int = 1) -> np.ndarray:
    """P^V_m(i) proportional to exp(x_m^T x_i / tau_v), each row normalised.  [N, N].

    With several images a row covers the tokens of its own image only
    (appendix "Appearance and spatial clients", last paragraphs).
    """
    logits = cos / p["tau_v"]
    if n_images > 1:
        img = image_index(cos.shape[0], n_images)
        logits = np.where(img[:, None] == img[None, :], logits, -np.inf)
    logits = logits - logits.max(axis=1, keepdims=True)
    E = np.exp(logits)
    return E / E.sum(axis=1, keepdims=True)


# ---------------------------------------------------------------------------
# Long prefixes: the bounded appearance bank (appendix "Appearance and spatial
# clients", last paragraph, and the cost paragraphs after Algorithm 1; Table
# "Shared GMC configuration", long-prefix row: rank 128, M_V <= 4096, b = 512)
# ---------------------------------------------------------------------------
def bounded_client_tokens(N: int, max_clients: int) -> np.ndarray:
    """The M_V = min(N, max_clients) uniformly spaced source tokens that act as
    appearance clients: c(m) = floor(m N / M_V), m = 0 .. M_V - 1 (every
    token when N <= max_clients)."""
    MV = min(N, max_clients)
    return (np.arange(MV, dtype=np.int64) * N) // MV


def projected_states(hvis: np.ndarray, R: np.ndarray, p: dict) -> np.ndarray:
    """Appearance states under the fixed rank-r Rademacher map R [r, D]:
    y_i = R h_i, x~_i = y_i / max(||y_i||, eps).  [N, r].  Normalising after
    the map makes x~ independent of R's scale (1 or 1/sqrt(r))."""
    y = hvis @ R.T
    n = np.sqrt(np.sum(y * y, axis=1))
    return y / np.maximum(n, p["norm_eps"])[:, None]


def bounded_appearance_clients(xt: np.ndarray, clients: np.ndarray, p: dict,
                               n_images: int = 1) -> np.ndarray:
    """Row m: P^V_m(i) proportional to exp(x~_{c(m)}^T x~_i / tau_v) over every
    token i of client c(m)'s image, normalised.  [M_V, N]."""
    logits = (xt[clients] @ xt.T) / p["tau_v"]
    if n_images > 1:
        img = image_index(xt.shape[0], n_images)
        logits = np.where(img[clients][:, None] == img[None, :], logits, -np.inf)
    logits = logits - logits.max(axis=1, keepdims=True)
    E = np.exp(logits)
    return E / E.sum(axis=1, keepdims=True)


def support_cosines(hvis: np.ndarray, S_sorted: np.ndarray, p: dict) -> np.ndarray:
    """cos(h_i, h_j) for every token i and selected j: [N, K], column k the
    k-th selected token (the N x K product the assignment needs)."""
    x = unit_states(hvis, p)
    return x @ x[np.asarray(S_sorted, dtype=np.int64)].T


def grid_coords(gh: int, gw: int) -> np.ndarray:
    """Normalised source coordinates p_i = ((r+0.5)/gh, (c+0.5)/gw), i = r*gw + c."""
    r, c = np.divmod(np.arange(gh * gw), gw)
    return np.stack([(r + 0.5) / gh, (c + 0.5) / gw], axis=1)


def landmark_coords(n: int) -> np.ndarray:
    """The n x n landmarks ((a+0.5)/n, (b+0.5)/n), l = a*n + b."""
    a, b = np.divmod(np.arange(n * n), n)
    return np.stack([(a + 0.5) / n, (b + 0.5) / n], axis=1)


def spatial_clients(gh: int, gw: int, p: dict, n_images: int = 1) -> np.ndarray:
    """P^S_l(i) proportional to 1[I_i = I_l] exp(-||p_i - l_l||^2 / tau_s), rows normalised.

    Every image has its own landmark grid in its normalised coordinates
    (Eq. (cond-aux-clients)): rows (image k, landmark l), k-major, each over
    image k's tokens.  [n_images * L^2, n_images * gh * gw].
    """
    P = grid_coords(gh, gw)
    Lm = landmark_coords(p["landmarks"])
    d2 = np.sum((Lm[:, None, :] - P[None, :, :]) ** 2, axis=2)
    logits = -d2 / p["tau_s"]
    logits = logits - logits.max(axis=1, keepdims=True)
    E = np.exp(logits)
    one = E / E.sum(axis=1, keepdims=True)
    if n_images == 1:
        return one
    L2, Ng = one.shape
    out = np.zeros((n_images * L2, n_images * Ng))
    for k in range(n_images):
        out[k * L2:(k + 1) * L2, k * Ng:(k + 1) * Ng] = one
    return out


# ---------------------------------------------------------------------------
# Client matrix (Eq. (cond-coverage)) and facility value (Eq. (3))
# ---------------------------------------------------------------------------
@dataclass
class ClientMatrix:
    C: np.ndarray                # [M, N] preweighted clients Cbar
    banks: dict                  # bank name -> slice of rows
    active: np.ndarray           # [M] active-row indicator a_m
    views: dict = None           # message view -> slice of its grounded rows


def client_matrix(PG, activeG, omega, nu, PV, PS, p) -> ClientMatrix:
    """Stack the three banks: rows (h, t) h-major, then appearance rows m, then landmarks l.

    Grounded row (h, t): beta_G * omega_h * nu_t * a_{h,t} * P^G_{h,t}.
    Appearance row m: (beta_V / M_V) P^V_m, M_V = N on the exact bank (every
    token a client) or the bounded bank's client count.  Spatial row l:
    (beta_S / M_S) P^S_l.
    """
    H, T, N = PG.shape
    MV = PV.shape[0]
    wG = p["beta_G"] * omega[:, None] * nu[None, :] * activeG
    G = (wG[:, :, None] * PG).reshape(H * T, N)
    V = (p["beta_V"] / MV) * PV
    S = (p["beta_S"] / PS.shape[0]) * PS
    C = np.concatenate([G, V, S], axis=0)
    banks = {"grounded": slice(0, H * T), "appearance": slice(H * T, H * T + MV),
             "spatial": slice(H * T + MV, H * T + MV + PS.shape[0])}
    active = np.concatenate([activeG.reshape(-1), np.ones(MV, bool), np.ones(PS.shape[0], bool)])
    return ClientMatrix(C, banks, active)


def client_matrix_views(PGs, actives, betas, omega, nu, PV, PS, p) -> ClientMatrix:
    """Eq. (cond-coverage) with message views: the grounded rows of every view
    (view v, h, t) h-major within the view, views in order (current first),
    then appearance rows, then landmarks.

    Grounded row (v, h, t): beta_v * omega_h * nu_t * a_{v,h,t} * P^G_{v,h,t}.
    The bank "grounded" spans every view's rows; ``views[v]`` each view's block.
    """
    blocks, act = [], []
    views = {}
    at = 0
    for v, (PG, a, beta) in enumerate(zip(PGs, actives, betas)):
        H, T, N = PG.shape
        w = beta * omega[:, None] * nu[None, :] * a
        blocks.append((w[:, :, None] * PG).reshape(H * T, N))
        act.append(a.reshape(-1))
        views[v] = slice(at, at + H * T)
        at += H * T
    MV = PV.shape[0]  # appearance clients (N on the exact bank)
    G = np.concatenate(blocks, axis=0)
    V = (p["beta_V"] / MV) * PV
    S = (p["beta_S"] / PS.shape[0]) * PS
    C = np.concatenate([G, V, S], axis=0)
    banks = {"grounded": slice(0, at), "appearance": slice(at, at + MV),
             "spatial": slice(at + MV, at + MV + PS.shape[0])}
    active = np.concatenate(act + [np.ones(MV, bool), np.ones(PS.shape[0], bool)])
    return ClientMatrix(C, banks, active, views)


def facility_value(C: np.ndarray, S) -> float:
    """F(S) = sum_m max_{i in S} C_mi, F(empty) = 0."""
    S = list(S)
    if not S:
        return 0.0
    return float(C[:, S].max(axis=1).sum())


# ---------------------------------------------------------------------------
# a8: batched responsibility selection (Eq. (4), Eq. (cond-responsibility))
# ---------------------------------------------------------------------------
def stable_top(values: np.ndarray, ids: np.ndarray, k: int) -> np.ndarray:
    """The k ids with the largest values, ties to the lowest id, in that order."""
    order = np.lexsort((ids, -values))
    return ids[order[:k]]


@dataclass
class SelectRound:
    gains: np.ndarray          # u_i for every token (0 for selected ones)
    own_pool: np.ndarray       # the oracle's pool
    pool: np.ndarray           # pool used (own or forced)
    scores: np.ndarray         # s over ``pool`` (aligned with it)
    own_batch: np.ndarray      # oracle's batch given ``pool``
    batch: np.ndarray          # batch used (own or forced)
    fill: bool                 # zero-gain fill round
    F_before: float
    F_after: float
    U: float                   # sum of the K largest remaining singleton gains
    seed: bool = False         # multi-image seed round: one max-gain token per image


@dataclass
class Selection:
    order: list                # indices in the order they entered S
    rounds: list = field(default_factory=list)
    K: int = 0

    @property
    def support(self) -> np.ndarray:
        return np.array(sorted(self.order), dtype=np.int64)


def select_support(C: np.ndarray, K: int, p: dict, forced=None, mode: str = "responsibility",
                   n_images: int = 1) -> Selection:
    """Deployed batched solver until |S| = K.

    Round t (support S_t, b_m = max_{j in S_t} C_mj, b = 0 for S empty):
      R = [C - b]_+,  u_i = sum_m R_mi;
      pool = top-min(pool_mult*b, #{u_i > 0}) unselected tokens by u;
      rho_m. = softmax over the pool of R_m. / (resp_temp * max_pool R_m. + eps);
      s_i = sum_m rho_mi R_mi;  the top-min(b, |pool|, K - |S|) pool tokens by s
      enter S together; then b is refreshed.
    Empty pool: the remaining budget is filled in ascending token order.
    mode="greedy" is exact sequential greedy (one token per round, argmax u),
    the special case used by the (1 - 1/e) guarantee.

    forced: optional list of (pool, batch) per round (a fill round has an
    empty pool and its filled tokens as batch).  When given, the oracle
    computes its own values, records them, then continues with the forced
    choice.

    n_images > 1: S starts with the token of largest singleton gain of every
    image (ties to the lowest index), recorded as a first "seed" round whose
    pool and batch are those tokens (Sec. 3.3; appendix "Batched
    complementary support"; Algorithm 1 step 3).
    """
    M, N = C.shape
    bsz = p["batch_b"] if mode == "responsibility" else 1
    pool_size = p["pool_mult"] * bsz
    selected = np.zeros(N, dtype=bool)
    bm = np.zeros(M)
    sel = Selection(order=[], K=K)
    ids = np.arange(N)
    rnd = 0
    if n_images > 1:
        u = C.sum(axis=0)  # S empty: every client value is a residual
        img = image_index(N, n_images)
        own = np.array([int(stable_top(u[img == k], ids[img == k], 1)[0]) for k in range(n_images)])
        f = forced[0] if forced is not None else None
        seeds = np.asarray(f[1], dtype=np.int64) if f is not None else own
        selected[seeds] = True
        sel.order.extend(int(i) for i in seeds)
        bm = C[:, seeds].max(axis=1)
        remaining = np.sort(u)[::-1]
        sel.rounds.append(SelectRound(u, own, own, u[own], own, seeds, False, 0.0,
                                      float(bm.sum()), float(remaining[:K].sum()), seed=True))
        rnd = 1
    while len(sel.order) < K:
        R = np.maximum(C - bm[:, None], 0.0)
        u = R.sum(axis=0)
        u[selected] = 0.0
        remaining = np.sort(u[~selected])[::-1]
        U = float(remaining[:K].sum())
        F0 = float(bm.sum())
        cand = ids[(~selected) & (u > 0)]
        own_pool = stable_top(u[cand], cand, pool_size) if cand.size else np.zeros(0, np.int64)
        f = forced[rnd] if forced is not None else None
        pool = np.asarray(f[0], dtype=np.int64) if f is not None else own_pool
        if pool.size == 0:
            need = K - len(sel.order)
            own_fill = ids[~selected][:need]
            batch = np.asarray(f[1], dtype=np.int64) if f is not None else own_fill
            selected[batch] = True
            sel.order.extend(int(i) for i in batch)
            bm = np.maximum(bm, C[:, batch].max(axis=1)) if batch.size else bm
            sel.rounds.append(SelectRound(u, own_pool, pool, np.zeros(0), own_fill, batch, True,
                                          F0, float(bm.sum()), U))
            rnd += 1
            continue
        RP = R[:, pool]
        if mode == "responsibility":
            rmax = RP.max(axis=1)
            logits = RP / (p["resp_temp"] * rmax + p["resp_eps"])[:, None]
            logits = logits - logits.max(axis=1, keepdims=True)
            rho = np.exp(logits)
            rho /= rho.sum(axis=1, keepdims=True)
            s = (rho * RP).sum(axis=0)
        else:
            s = u[pool].copy()
        nb = min(bsz, pool.size, K - len(sel.order))
        own_batch = stable_top(s, pool, nb)
        batch = np.asarray(f[1], dtype=np.int64) if f is not None else own_batch
        selected[batch] = True
        sel.order.extend(int(i) for i in batch)
        bm = np.maximum(bm, C[:, batch].max(axis=1))
        sel.rounds.append(SelectRound(u, own_pool, pool, s, own_batch, batch, False,
                                      F0, float(bm.sum()), U))
        rnd += 1
    return sel


def batched_certificate(sel: Selection) -> float:
    """c_B = 1 - prod_t (1 - q_t), q_t = [F(S_t u B_t) - F(S_t)] / U_t over rounds with U_t > 0.

    Eq. (6) / Eq. (cond-batched-bound).
    """
    prod = 1.0
    for r in sel.rounds:
        if r.U > 0:
            prod *= 1.0 - (r.F_after - r.F_before) / r.U
    return 1.0 - prod


def bank_saturation(cm: ClientMatrix, S):
    """c_b(S) = F_b(S) / F_b(V), omega_b = Z_b / sum_c Z_c (Eq. (cond-saturation)).

    Returns dict bank -> (F_b(S), Z_b = F_b(V), omega_b).
    """
    N = cm.C.shape[1]
    out = {}
    Z = {b: facility_value(cm.C[s], range(N)) for b, s in cm.banks.items()}
    tot = sum(Z.values())
    for b, s in cm.banks.items():
        out[b] = (facility_value(cm.C[s], S), Z[b], Z[b] / tot if tot > 0 else 0.0)
    return out


# ---------------------------------------------------------------------------
# a9: population assignment (Eq. (cond-assignment), (cond-population-gate))
# ---------------------------------------------------------------------------
@dataclass
class Assignment:
    pi: np.ndarray             # [N] representative of each token
    delta: np.ndarray          # [N] best minus second-best selected cosine (0 for selected)
    delta_bar: float
    s_x: float
    g: np.ndarray              # [N] local ambiguity gate
    kappa_best: np.ndarray     # [N] max_j kappa_ij (discarded tokens)
    kappa_chosen: np.ndarray   # [N] kappa at the assignment used


def assign_population(cos: np.ndarray, S: np.ndarray, gh: int, gw: int, p: dict,
                      forced_pi=None, n_images: int = 1, support_cols: bool = False) -> Assignment:
    """pi(i) = argmax_{j in S} cos_ij + lambda_p s_x g_i exp(-||p_i - p_j||^2 / tau_s).

    Selected tokens represent themselves.  delta_i is the gap between the
    largest and second-largest selected cosine (0 when |S| = 1); Delta_bar is
    its mean over discarded tokens (0 when none is discarded);
    s_x = 1 - exp[-(Delta_bar / gate_scale)^gate_pow];
    g_i = exp[-(delta_i / ambig_margin)^gate_pow].  Ties go to the lowest j.
    With several images, token i's candidates S_i are the selected tokens of
    its own image, and both the gap and the coordinates are within that image.
    support_cols: ``cos`` is [N, |S|], column k holding the cosines with the
    k-th token of S (``support_cosines``), instead of [N, N].
    """
    N = cos.shape[0]
    S = np.asarray(S, dtype=np.int64)
    if support_cols:
        colof = {int(j): k for k, j in enumerate(S)}
        cos_at = lambda i, js: cos[i, [colof[int(j)] for j in js]]  # noqa: E731
    else:
        cos_at = lambda i, js: cos[i, js]  # noqa: E731
    in_S = np.zeros(N, bool)
    in_S[S] = True
    disc = np.flatnonzero(~in_S)
    img = image_index(N, n_images)
    compat = {int(i): S[img[S] == img[i]] for i in disc}  # S_i: same-image carriers
    delta = np.zeros(N)
    for i in disc:
        v = np.sort(cos_at(i, compat[int(i)]))[::-1]
        delta[i] = v[0] - v[1] if v.size > 1 else 0.0
    delta_bar = float(delta[disc].mean()) if disc.size else 0.0
    s_x = 1.0 - math.exp(-((delta_bar / p["gate_scale"]) ** p["gate_pow"]))
    g = np.exp(-((delta / p["ambig_margin"]) ** p["gate_pow"]))
    P = np.tile(grid_coords(gh, gw), (n_images, 1))  # coordinates in each token's own grid
    pi = np.arange(N)
    kb = np.zeros(N)
    kc = np.zeros(N)
    for i in disc:
        Si = compat[int(i)]
        d2 = np.sum((P[Si] - P[i]) ** 2, axis=1)
        kappa = cos_at(i, Si) + p["assign_spatial_w"] * s_x * g[i] * np.exp(-d2 / p["tau_s"])
        j = int(stable_top(kappa, Si, 1)[0])
        pi[i] = j if forced_pi is None else int(forced_pi[i])
        kb[i] = kappa.max()
        hit = np.flatnonzero(Si == pi[i])
        kc[i] = kappa[hit[0]] if hit.size else -np.inf
    if forced_pi is not None:
        pi[S] = np.asarray(forced_pi)[S]
    return Assignment(pi, delta, delta_bar, s_x, g, kb, kc)


# ---------------------------------------------------------------------------
# a10: transport (Eq. (5), Eq. (cond-transport))
# ---------------------------------------------------------------------------
def population_weights(ebar: np.ndarray, s_x: float, p: dict) -> np.ndarray:
    """m_i = (1 - alpha s_x) + alpha s_x ebar_i (Eq. (cond-population-gate))."""
    a = p["pop_strength"]
    return (1.0 - a * s_x) + a * s_x * ebar


def rms(u: np.ndarray, axis=-1):
    return np.sqrt(np.mean(u * u, axis=axis))


@dataclass
class Transport:
    mass: np.ndarray            # [K] M_j, aligned with the sorted support
    centroid: np.ndarray        # [K, D] c_j
    restored: np.ndarray        # [K, D] R_j(c_j)


def transport(hvis: np.ndarray, S_sorted: np.ndarray, pi: np.ndarray, m: np.ndarray, p: dict) -> Transport:
    """M_j = sum_{pi(i)=j} m_i, c_j = M_j^-1 sum m_i h_i, h~_j = c_j rms(h_j) / (rms(c_j) + eps)."""
    K = S_sorted.size
    D = hvis.shape[1]
    slot = {int(j): k for k, j in enumerate(S_sorted)}
    Msum = np.zeros(K)
    acc = np.zeros((K, D))
    for i in range(hvis.shape[0]):
        k = slot[int(pi[i])]
        Msum[k] += m[i]
        acc[k] += m[i] * hvis[i]
    c = acc / Msum[:, None]
    scale = rms(hvis[S_sorted]) / (rms(c) + p["rms_eps"])
    return Transport(Msum, c, c * scale[:, None])


# ---------------------------------------------------------------------------
# a11: physical compaction (Algorithm 1 step 6; index map)
# ---------------------------------------------------------------------------
def compaction_rows(S_sorted: np.ndarray, N: int, T: int) -> np.ndarray:
    """Source sequence rows kept, in order: selected visual rows ascending, then all text rows."""
    return np.concatenate([np.asarray(S_sorted, dtype=np.int64), N + np.arange(T)])


def gather_prefix_kv(prefix, rows: np.ndarray):
    """Cached path: the dense K/V of prefix layers 0..p-1 at the kept sequence rows.

    Appendix "Index map and physical token accounting": the prompt K/V of the
    blocks before the boundary are gathered, unchanged, at the retained
    sequence indices (selected visual rows ascending, then every text row);
    only layers from the boundary on see transported states.  `prefix` lists
    (K_l, V_l), each [N+T, Hkv, d]; returns [p, 2, len(rows), Hkv, d].
    """
    if not prefix:
        return np.zeros((0, 2, rows.size, 0, 0))
    return np.stack([np.stack([K_l[rows], V_l[rows]]) for K_l, V_l in prefix])


# ---------------------------------------------------------------------------
# Whole step (Algorithm 1, steps 2-6) for one image
# ---------------------------------------------------------------------------
@dataclass
class Result:
    K: int
    identity: bool
    A: np.ndarray = None
    Z: np.ndarray = None
    sigma: np.ndarray = None
    unorm: np.ndarray = None
    PG: np.ndarray = None
    activeG: np.ndarray = None
    nu: np.ndarray = None
    heads: HeadClusters = None
    e: np.ndarray = None
    ebar: np.ndarray = None
    cos: np.ndarray = None
    clients: ClientMatrix = None
    selection: Selection = None
    support: np.ndarray = None
    assignment: Assignment = None
    m: np.ndarray = None
    transport: Transport = None
    rows: np.ndarray = None        # source rows of the compact sequence
    out_hidden: np.ndarray = None  # float64 compact hidden (transported visual rows, text rows)
    out_kv: np.ndarray = None      # [2, K+T, Hkv, d]
    out_pos: np.ndarray = None     # [3, K+T]
    out_prefix_kv: np.ndarray = None  # [p, 2, K+T, Hkv, d] dense prefix layers at the kept rows
    history: list = None           # per historical view: (A, Z, sigma, unorm, PG, active)
    xt: np.ndarray = None          # long prefixes: projected appearance states [N, r]
    clients_V: np.ndarray = None   # long prefixes: tokens of the appearance clients [M_V]
    cos_support: np.ndarray = None  # long prefixes: support cosines [N, K]


def compress(hidden, Kall, Vall, Q, pos, W, gh, gw, K_r, p=None, forced=None,
             history=None, prefix=None, n_images: int = 1, long_prefix=None) -> Result:
    """Grounded Message Coreset compression of one image boundary.

    hidden [N+T, D], Kall/Vall [N+T, Hkv, d], Q [T, H, d], pos [3, N+T],
    W [H, d, r].  ``forced`` may hold "centres", "head_assign", "rounds",
    "pi" to follow choices made elsewhere (see the module docstring).
    ``history`` (optional) lists completed historical message views, each a
    dict with that layer's text queries "Q" [T, H, d], keys "K" and values
    "V" [N+T, Hkv, d] and probe "W" [H, d, r] (Appendix "Native message
    clients"): every view adds its own grounded rows, the head patterns span
    all views, the views share beta_hist equally, and the message energy stays
    the current view's (Eq. (cond-grounded-energy)).
    ``n_images`` > 1: a multi-image prompt whose visual segment holds that many
    images of gh x gw tokens one after another (budget, seeds, banks and
    assignment per image as the paper states; see the functions above).
    ``prefix`` (optional) lists the dense prefix layers' (K, V), each
    [N+T, Hkv, d]; ``out_prefix_kv`` then holds them at the kept rows
    (``gather_prefix_kv``).
    ``long_prefix`` (optional) selects the bounded appearance bank of long
    prefixes: a dict with the Rademacher map "R" [r, D] and "max_clients".
    The appearance clients are then the uniformly spaced tokens of
    ``bounded_client_tokens`` over the projected states, and the assignment
    reads only the N x K support cosines (``support_cosines``); ``cos`` is
    None and ``cos_support`` holds them.  The responsibility batch b comes
    from ``p`` as always (the long-prefix row of the configuration table uses
    b = 512).
    """
    p = p or params()
    forced = forced or {}
    N = gh * gw * n_images
    T, H, d = Q.shape
    K = budget(K_r, N, n_images)
    if K == N:   # K = N returns the unmodified execution
        rows = np.arange(N + T)
        return Result(K=K, identity=True, support=np.arange(N), rows=rows,
                      out_hidden=np.array(hidden, dtype=np.float64),
                      out_kv=np.stack([Kall, Vall]), out_pos=np.array(pos),
                      out_prefix_kv=gather_prefix_kv(prefix, rows))
    res = Result(K=K, identity=False)
    hvis = hidden[:N]
    res.A = message_slice(Q, Kall, N)
    res.Z, res.sigma = probe_values(Vall[:N], W, H, p)
    res.unorm = atom_norms(res.A, res.Z, res.sigma)
    res.PG, res.activeG = grounded_clients(res.unorm)
    res.nu = query_weights(T, p)
    views = None
    if history is not None:
        res.history = []
        views = [(res.A, res.Z, res.sigma, p["beta_G"])]
        for view in history:
            A_v = message_slice(view["Q"], view["K"], N)
            Z_v, s_v = probe_values(view["V"][:N], view["W"], H, p)
            un_v = atom_norms(A_v, Z_v, s_v)
            PG_v, act_v = grounded_clients(un_v)
            res.history.append((A_v, Z_v, s_v, un_v, PG_v, act_v))
            views.append((A_v, Z_v, s_v, p["beta_hist"] / len(history)))
    res.heads = head_clusters(res.A, res.Z, res.sigma, p,
                              forced.get("centres"), forced.get("head_assign"), views=views)
    res.e, res.ebar = message_energy(res.unorm, res.heads.omega, res.nu)
    if long_prefix is None:
        res.cos = cosine_matrix(hvis, p)
        PV = appearance_clients(res.cos, p, n_images)
    else:
        res.xt = projected_states(hvis, np.asarray(long_prefix["R"], dtype=np.float64), p)
        res.clients_V = bounded_client_tokens(N, int(long_prefix["max_clients"]))
        PV = bounded_appearance_clients(res.xt, res.clients_V, p, n_images)
    PS = spatial_clients(gh, gw, p, n_images)
    if history is None:
        res.clients = client_matrix(res.PG, res.activeG, res.heads.omega, res.nu, PV, PS, p)
    else:
        res.clients = client_matrix_views(
            [res.PG] + [hv[4] for hv in res.history], [res.activeG] + [hv[5] for hv in res.history],
            [v[3] for v in views], res.heads.omega, res.nu, PV, PS, p)
    res.selection = select_support(res.clients.C, K, p, forced=forced.get("rounds"),
                                   n_images=n_images)
    res.support = res.selection.support
    if long_prefix is None:
        res.assignment = assign_population(res.cos, res.support, gh, gw, p, forced.get("pi"),
                                           n_images)
    else:
        res.cos_support = support_cosines(hvis, res.support, p)
        res.assignment = assign_population(res.cos_support, res.support, gh, gw, p,
                                           forced.get("pi"), n_images, support_cols=True)
    res.m = population_weights(res.ebar, res.assignment.s_x, p)
    res.transport = transport(hvis, res.support, res.assignment.pi, res.m, p)
    res.rows = compaction_rows(res.support, N, T)
    res.out_hidden = np.concatenate([res.transport.restored, hidden[N:]], axis=0)
    res.out_kv = np.stack([Kall[res.rows], Vall[res.rows]])
    res.out_pos = np.asarray(pos)[:, res.rows]
    res.out_prefix_kv = gather_prefix_kv(prefix, res.rows)
    return res
