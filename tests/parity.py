"""GPU <-> oracle comparison helpers.

The CUDA path and the fp64 oracle make the same discrete choices (head
centres, pool, batch, assignment) from values computed in different
precisions.  A choice is checked against the oracle's fp64 values: it must be
a valid top-k (or argmax) of those values up to a relative margin TOL = 1e-4
of the largest value.  Where the margin between the k-th and (k+1)-th value
exceeds TOL the valid choice is unique, so the kept indices are then
bit-exact; inside the margin either side of a near-tie is accepted and the
oracle follows the GPU's choice (``forced``) so one tie cannot cascade.
"""

from __future__ import annotations

import ctypes
from dataclasses import dataclass, field

import numpy as np

from oracle import gmc_oracle as O

TOL = 1e-4


@dataclass
class Decisions:
    checked: int = 0
    exact: int = 0
    near_ties: list = field(default_factory=list)
    failures: list = field(default_factory=list)

    def ok(self):
        return not self.failures


def valid_topk(values: np.ndarray, ids: np.ndarray, chosen, k: int, tol: float = TOL):
    """Is ``chosen`` a valid set of the k largest ``values`` (aligned with ``ids``) up to tol?

    Returns (valid, exact): exact when it equals the stable top-k.
    """
    chosen = np.asarray(sorted(int(c) for c in chosen), dtype=np.int64)
    if chosen.size != k or len(set(chosen.tolist())) != k:
        return False, False
    order = np.lexsort((ids, -values))
    top = np.sort(ids[order[:k]])
    if np.array_equal(top, chosen):
        return True, True
    if k == 0:
        return True, True
    scale = max(float(np.max(np.abs(values))), 1e-300)
    cut = float(values[order[k - 1]])
    pos = {int(i): n for n, i in enumerate(ids)}
    if any(int(c) not in pos for c in chosen):
        return False, False
    inset = np.zeros(ids.size, bool)
    inset[[pos[int(c)] for c in chosen]] = True
    must_in = values > cut + tol * scale
    must_out = values < cut - tol * scale
    return bool(np.all(inset[must_in]) and not np.any(inset[must_out])), False


# ---------------------------------------------------------------------------
# Trace parsing (layout from gmc_get_trace_layout)
# ---------------------------------------------------------------------------
class TraceHeaderNP(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int32), ("rounds", ctypes.c_int32), ("n_clusters", ctypes.c_int32),
                ("filled", ctypes.c_int32), ("s_x", ctypes.c_float), ("delta_bar", ctypes.c_float),
                ("F_S", ctypes.c_float * 3), ("F_V", ctypes.c_float * 3), ("c_B", ctypes.c_float),
                ("reserved", ctypes.c_int32 * 3)]


@dataclass
class ImageTrace:
    K: int
    rounds: int
    n_clusters: int
    filled: int
    s_x: float
    delta_bar: float
    F_S: list
    F_V: list
    c_B: float
    order: np.ndarray
    round_end: np.ndarray
    pool: np.ndarray
    centres: np.ndarray
    head_assign: np.ndarray
    omega: np.ndarray
    pi: np.ndarray
    ebar: np.ndarray
    mass: np.ndarray

    def forced_rounds(self):
        """[(pool, batch)] per round as the oracle's ``forced`` argument takes them."""
        out, prev = [], 0
        for t in range(self.rounds):
            end = int(self.round_end[t])
            pool = self.pool[t][self.pool[t] >= 0]
            out.append((pool, self.order[prev:end]))
            prev = end
        return out


def parse_trace(buf: np.ndarray, layout, B: int, K: int, H: int, N: int, max_clusters: int = 4):
    raw = np.asarray(buf, dtype=np.uint8)
    out = []
    for b in range(B):
        rec = raw[b * layout.bytes_per_image:(b + 1) * layout.bytes_per_image]
        hd = TraceHeaderNP.from_buffer_copy(rec[:ctypes.sizeof(TraceHeaderNP)].tobytes())

        def arr(off, n, dt):
            return rec[off:off + 4 * n].view(dt).copy()

        R, P = layout.rounds_max, layout.pool_size
        out.append(ImageTrace(
            hd.K, hd.rounds, hd.n_clusters, hd.filled, hd.s_x, hd.delta_bar, list(hd.F_S), list(hd.F_V),
            hd.c_B,
            arr(layout.off_order, K, np.int32), arr(layout.off_round_end, R, np.int32),
            arr(layout.off_pool, R * P, np.int32).reshape(R, P),
            arr(layout.off_centres, max_clusters, np.int32), arr(layout.off_head_assign, H, np.int32),
            arr(layout.off_omega, H, np.float32), arr(layout.off_pi, N, np.int32),
            arr(layout.off_ebar, N, np.float32), arr(layout.off_mass, N, np.float32)))
    return out


# ---------------------------------------------------------------------------
# Decision checks
# ---------------------------------------------------------------------------
def check_selection(sel: O.Selection, P: int, dec: Decisions, tag=""):
    """Every forced round against the oracle's fp64 gains and scores."""
    if not sel.rounds:
        return
    N = sel.rounds[0].gains.size
    scale0 = max(float(sel.rounds[0].gains.max()), 1e-300)
    selected = np.zeros(N, bool)
    for t, r in enumerate(sel.rounds):
        u = r.gains
        free = np.flatnonzero(~selected)
        dec.checked += 1
        if getattr(r, "seed", False):
            # multi-image seed round: every image's token of largest singleton gain
            I = len(r.batch)
            Ng = N // I
            for k, jk in enumerate(np.asarray(r.batch)):
                ids = np.arange(k * Ng, (k + 1) * Ng)
                ok, exact = valid_topk(u[ids], ids, [int(jk)], 1)
                if not ok:
                    dec.failures.append(f"{tag} seed of image {k}: {int(jk)} is not its best gain")
                elif not exact:
                    dec.near_ties.append(f"{tag} seed of image {k}")
            dec.exact += 1
            selected[r.batch] = True
            continue
        if r.fill:
            # valid only when every remaining gain is (near) zero; ascending order
            if u[free].max(initial=0.0) > TOL * scale0:
                dec.failures.append(f"{tag} round {t}: fill while gains are positive")
            elif not np.array_equal(np.asarray(r.batch), free[:len(r.batch)]):
                dec.failures.append(f"{tag} round {t}: fill not in ascending order")
            elif r.own_pool.size == 0:
                dec.exact += 1
            else:
                dec.near_ties.append(f"{tag} round {t}: fill over near-zero gains")
            selected[r.batch] = True
            continue
        k = r.pool.size
        ok, exact = valid_topk(u[free], free, r.pool, k)
        npos = int(np.sum(u[free] > 0))
        if k != min(P, npos):
            srt = np.sort(u[free])[::-1]
            cut = srt[k] if k < srt.size else 0.0
            ok = ok and cut <= TOL * scale0
            exact = False
        if not ok:
            dec.failures.append(f"{tag} round {t}: pool outside the {TOL} margin")
        elif exact:
            dec.exact += 1
        else:
            dec.near_ties.append(f"{tag} round {t}: pool")
        nb = len(r.batch)
        ok, exact = valid_topk(r.scores, r.pool, r.batch, nb)
        dec.checked += 1
        if not ok:
            dec.failures.append(f"{tag} round {t}: batch outside the {TOL} margin "
                                f"(gpu {sorted(np.asarray(r.batch).tolist())} oracle {sorted(r.own_batch.tolist())})")
        elif exact:
            dec.exact += 1
        else:
            dec.near_ties.append(f"{tag} round {t}: batch")
        selected[r.batch] = True


def check_heads(hc: O.HeadClusters, dec: Decisions, tag=""):
    H = hc.cos.shape[0]
    c = hc.centres
    dec.checked += 1
    vals = hc.pre_norm
    ok, exact = valid_topk(vals, np.arange(H), [c[0]], 1)
    if not ok:
        dec.failures.append(f"{tag} first head centre {c[0]}")
    elif exact:
        dec.exact += 1
    else:
        dec.near_ties.append(f"{tag} first centre")
    for n in range(1, len(c)):
        rest = np.array([h for h in range(H) if h not in c[:n]])
        mc = np.array([max(hc.cos[h, cc] for cc in c[:n]) for h in rest])
        ok, exact = valid_topk(-mc, rest, [c[n]], 1)
        dec.checked += 1
        if not ok:
            dec.failures.append(f"{tag} head centre {n}")
        elif exact:
            dec.exact += 1
        else:
            dec.near_ties.append(f"{tag} centre {n}")
    for h in range(H):
        sims = np.array([hc.cos[h, cc] for cc in c])
        ok, exact = valid_topk(sims, np.arange(len(c)), [hc.assign[h]], 1)
        dec.checked += 1
        if not ok:
            dec.failures.append(f"{tag} head {h} cluster")
        elif exact:
            dec.exact += 1
        else:
            dec.near_ties.append(f"{tag} head {h} cluster")


def check_assignment(a: O.Assignment, S: np.ndarray, dec: Decisions, tag=""):
    N = a.pi.size
    inS = np.zeros(N, bool)
    inS[S] = True
    if not np.all(a.pi[S] == S):
        dec.failures.append(f"{tag} a selected token does not represent itself")
    for i in np.flatnonzero(~inS):
        dec.checked += 1
        best, got = a.kappa_best[i], a.kappa_chosen[i]
        if got < best - TOL * max(1.0, abs(best)):
            dec.failures.append(f"{tag} token {i}: kappa {got:.6f} < best {best:.6f}")
        elif got == best:
            dec.exact += 1
        else:
            dec.near_ties.append(f"{tag} token {i} assignment")


def rel_row_err(gpu: np.ndarray, ref: np.ndarray) -> float:
    """max over rows of max|gpu - ref| / max|ref| (row-normalised max error)."""
    num = np.max(np.abs(gpu - ref), axis=1)
    den = np.maximum(np.max(np.abs(ref), axis=1), 1e-30)
    return float(np.max(num / den)) if num.size else 0.0
