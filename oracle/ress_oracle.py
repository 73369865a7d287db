"""ReSS oracle in float64 (test infrastructure: only the tests, the smoke check and the
benchmark's CPU baseline use it; nothing in the product path imports it).

Notation follows the paper: heads h, query block i, key block j, pooled probability
P_ij (Sec. 4.1), pooled value V_j, dense pooled output v_bar_i (Eq. 1), candidate set
cal_P (key blocks made only of patch tokens), keep budget c_h, drop set D, deviation
e_ij = v_bar_i - V_j, drift contribution d_ij = P_ij e_ij (Eq. 5), head slice W_O^h of
the output projection, block drift score s_ij (Eq. 6), cut key (Eq. 7), net drift g and
remaining mass K (Eq. 10), objective J = G / K^2 (Eq. 12), swap schedule m_r (Eq. 17).

Readings where the paper is silent:
  * Pooling: Q, K and V are mean-pooled over the valid tokens of each 64-token block; the
    pooled logits are q_bar_i . k_bar_j / sqrt(d_h) and P_i is their softmax over all key
    blocks (Sec. 3 step (1), Sec. 4.1).
  * Special tokens sit at the end of the sequence.  Key blocks that contain any of them
    form B minus cal_P and are always kept; query blocks that contain any of them are
    computed densely and carry no objective (Sec. 3, Sec. 4.1).
  * The same clamp max(., eps), eps = 1e-4, that Eq. 7 puts on 1 - P guards every
    remaining-mass denominator, so that J({j}) equals the squared Eq. 7 key (Sec. 4.3).
  * m_r = floor(rho c_h / 2^(r+1)), clamped to min(|D|, |cal_P \\ D|); m_r = 0 leaves the
    round a no-op (Eq. 17 gives a real number).
  * Each round chooses its restores and its drops from the same round-start state (one
    gain evaluation per round, Sec. 4.3 and Appendix E), then recomputes g, K and J of the
    new set by definition; track-best keeps the first set reaching the smallest J
    (strict <, Sec. 4.3 / Appendix B.3).
  * Every top-k orders by (value descending, block index ascending).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

EPS = 1e-4          # epsilon of Eq. 7
BLOCK = 64          # query and key block size of the 64x64 block grid
NEAR_THRESHOLD = 1e-3   # rows whose smallest decision margin is below this are "near-threshold"


# ----------------------------------------------------------------------------------------
# shapes
# ----------------------------------------------------------------------------------------
def n_blocks(n_tokens: int, block: int = BLOCK) -> int:
    """Number of blocks of the sequence; the last one may be partial."""
    return -(-n_tokens // block)


def n_candidates(n_tokens: int, n_special: int, block: int = BLOCK) -> int:
    """|cal_P|: blocks holding patch tokens only (special tokens are the trailing ones)."""
    return (n_tokens - n_special) // block


def swap_schedule(c: int, rounds: int, rho: float) -> list[int]:
    """Eq. 17: m_r = rho 2^-(r+1) c_h for r = 0..R-1, rounded down to a whole block count."""
    return [int(math.floor(float(rho) * c / float(2 ** (r + 1)))) for r in range(rounds)]


def top_m(values: np.ndarray, m: int) -> np.ndarray:
    """Positions of the m largest values, ordered by (value desc, position asc)."""
    order = sorted(range(values.size), key=lambda k: (-values[k], k))
    return np.array(order[:m], dtype=np.int64)


def ranked(values: np.ndarray) -> np.ndarray:
    """All values sorted by (value desc, position asc)."""
    order = sorted(range(values.size), key=lambda k: (-values[k], k))
    return values[np.array(order, dtype=np.int64)] if values.size else values


# ----------------------------------------------------------------------------------------
# Sec. 3 step (1) and Sec. 4.1: block pooling and the pooled attention map
# ----------------------------------------------------------------------------------------
def pool_blocks(X: np.ndarray, block: int = BLOCK) -> np.ndarray:
    """Mean over the valid tokens of each block.  X: [N, H, d] -> [H, nb, d] float64."""
    N, H, d = X.shape
    nb = n_blocks(N, block)
    out = np.empty((H, nb, d), dtype=np.float64)
    for j in range(nb):
        seg = np.asarray(X[j * block: min(N, (j + 1) * block)], dtype=np.float64)
        out[:, j, :] = seg.sum(axis=0) / seg.shape[0]
    return out


def pooled_attention_row(qbar_i: np.ndarray, Kb_h: np.ndarray) -> np.ndarray:
    """P_i. = softmax over all key blocks j in B of q_bar_i . k_bar_j / sqrt(d_h) (Sec. 4.1)."""
    d = qbar_i.shape[-1]
    logits = (Kb_h @ qbar_i) / math.sqrt(d)
    z = np.exp(logits - logits.max())
    return z / z.sum()


def dense_pooled_output(P_i: np.ndarray, Vb_h: np.ndarray) -> np.ndarray:
    """Eq. 1: v_bar_i = sum_{j in B} P_ij V_j."""
    return P_i @ Vb_h


def head_projection(W_o: np.ndarray, h: int, d_h: int) -> np.ndarray:
    """W_O^h in R^{d x d_h}: the columns of the output projection (Linear.weight, out x in)
    that multiply head h's output."""
    return np.asarray(W_o[:, h * d_h:(h + 1) * d_h], dtype=np.float64)


# ----------------------------------------------------------------------------------------
# Sec. 4.2: drift contributions, block drift score, cut key
# ----------------------------------------------------------------------------------------
def residual_contributions(P_i: np.ndarray, vbar_i: np.ndarray, Vb_h: np.ndarray,
                           WOh: np.ndarray):
    """Eq. 5 and Eq. 6 with the per-pair residual-space vector formed explicitly.

    Returns e [nb, d_h] (e_ij = v_bar_i - V_j), d [nb, d_h] (d_ij = P_ij e_ij) and
    r [nb, d] (r_ij = W_O^h d_ij, the (n_h, q_blk, k_blk, d) intermediate of Sec. 4.2).
    """
    e = vbar_i[None, :] - Vb_h
    dvec = P_i[:, None] * e
    r = dvec @ WOh.T
    return e, dvec, r


def drift_scores(r: np.ndarray) -> np.ndarray:
    """Eq. 6: s_ij = ||W_O^h d_ij||_2."""
    return np.sqrt((r * r).sum(axis=1))


def cut_keys(s: np.ndarray, P_i: np.ndarray) -> np.ndarray:
    """Eq. 7: s_ij / max(1 - P_ij, eps)."""
    return s / np.maximum(1.0 - P_i, EPS)


# ----------------------------------------------------------------------------------------
# Sec. 4.3: objective of a drop set, restoration rounds
# ----------------------------------------------------------------------------------------
def objective(D: np.ndarray, P_i: np.ndarray, r: np.ndarray):
    """Eq. 10-12 for the drop set D (boolean over the key blocks).

    g = sum_{j in D} d_ij is carried through W_O^h as a = W_O^h g = sum_{j in D} r_ij;
    K = 1 - sum_{j in D} P_ij; G = g^T M_h g = ||a||^2; J = G / max(K, eps)^2.
    Returns (J, a, K).
    """
    a = r[D].sum(axis=0) if D.any() else np.zeros(r.shape[1])
    K = 1.0 - P_i[D].sum()
    G = float(a @ a)
    return G / max(K, EPS) ** 2, a, K


def round_gains(D: np.ndarray, n_cand: int, P_i: np.ndarray, r: np.ndarray,
                J: float, a: np.ndarray, K: float):
    """Eq. 13-16 by direct recomputation from the round-start state.

    Restoring k in D gives g - d_ik, K + P_ik (Eq. 13); dropping a kept candidate k gives
    g + d_ik, K - P_ik.  The gain is the exact decrease of J (Eq. 16).  Returns the
    restore candidates, their gains, the drop candidates and their gains.
    """
    inD = np.nonzero(D[:n_cand])[0]
    outD = np.nonzero(~D[:n_cand])[0]
    a_res = a[None, :] - r[inD]
    J_res = (a_res * a_res).sum(axis=1) / np.maximum(K + P_i[inD], EPS) ** 2
    a_drop = a[None, :] + r[outD]
    J_drop = (a_drop * a_drop).sum(axis=1) / np.maximum(K - P_i[outD], EPS) ** 2
    return inD, J - J_res, outD, J - J_drop


def _gap(vals_sorted: np.ndarray, m: int, floor: float) -> float:
    """Decision margin of a top-m cut: the gap between the m-th and (m+1)-th entries of a
    descending list, relative to the larger magnitude of the two (at least `floor`); inf when
    the list has no (m+1)-th entry or m is 0 (nothing is decided)."""
    if m <= 0 or m >= vals_sorted.size:
        return math.inf
    a, b = vals_sorted[m - 1], vals_sorted[m]
    scale = max(abs(a), abs(b), floor)
    return (a - b) / scale if scale > 0 else 0.0


def _track_margin(J: float, J_best: float) -> float:
    """Decision margin of a track-best comparison (Sec. 4.3, Appendix B.3): how far the new
    objective J is from the best one so far, relative to that best (inf when J_best is 0)."""
    return abs(J - J_best) / J_best if J_best > 0 else math.inf


def _cdf_margins(masses, tau: float, keys_sorted: np.ndarray, n_add: int) -> list:
    """Decision margins of the CDF threshold: every running kept mass that was compared with
    tau, relative to tau, and the key gaps on both sides of the last block that joined (a
    swap there changes which blocks cross the threshold)."""
    out = [abs(x - tau) / tau for x in masses]
    if keys_sorted.size:
        out += [_gap(keys_sorted, n_add, 0.0), _gap(keys_sorted, n_add - 1, 0.0)]
    return out


@dataclass
class RowSelection:
    """ReSS result for one (head h, query block i) row."""
    h: int
    i: int
    dense: bool
    D0: np.ndarray            # initial drop set (bool over key blocks)
    D_best: np.ndarray        # returned drop set (track-best)
    J0: float
    J_best: float
    J_trace: list = field(default_factory=list)   # J of the current set after each round
    margin: float = math.inf  # smallest relative decision margin of the row
    swaps: int = 0            # sum of the m actually applied
    # every decision margin of the row in the order taken: ("cut", value) for the Eq. 7 cut,
    # ("cdf", value) for the CDF threshold, ("restore", r, value) / ("drop", r, value) for the
    # top-m cuts of round r and ("track", r, value) for its track-best comparison
    margins: list = field(default_factory=list)

    def note(self, kind: str, value: float, r: int = None) -> None:
        """Record one decision margin and keep the row's smallest."""
        self.margins.append((kind, value) if r is None else (kind, r, value))
        self.margin = min(self.margin, value)

    @property
    def near_threshold(self) -> bool:
        return self.margin < NEAR_THRESHOLD

    def kept(self) -> np.ndarray:
        """Selected blocks plus the always-kept ones, ascending (Sec. 3 step (3))."""
        return np.nonzero(~self.D_best)[0].astype(np.int32)


@dataclass(frozen=True)
class Variant:
    """Selection variants of the paper's ablations (Sec. 6: Fig. 8's sign flip, Table 3's
    probability selection; the random baseline of Fig. 8).

    key:      "drift" (Eq. 7, ReSS), "probability" (the pooled P_ij alone: top-k by attention
              mass, the rule of the probability-based methods) or "random" (SplitMix64 of a
              counter, see random_keys).
    maximize: "none" (ReSS minimises the drift), "swap" (restoration maximises J, the initial
              selection is unchanged) or "full" (the initial selection keeps the c_h smallest
              keys and restoration maximises J).
    cdf:      0 (off) or a threshold tau in (0, 1]: the CDF threshold of Table 3 (the top-p
              rule of probability-based selection on the pooled map).  Beyond its c_h
              top-key candidates a row keeps further candidates, in key order (value desc,
              index asc), until the pooled mass of its kept blocks, the always-kept ones
              included, reaches tau.  Defined without restoration rounds.
    """
    key: str = "drift"
    maximize: str = "none"
    seed: int = 0
    cdf: float = 0.0


RESS = Variant()
_MASK64 = (1 << 64) - 1


def splitmix64(x: int) -> int:
    """SplitMix64 (Steele, Lea and Flood, OOPSLA 2014): the state advanced by the golden-ratio
    increment, then the variant-13 mix of that paper.  Returns the output for state x."""
    z = (x + 0x9E3779B97F4A7C15) & _MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK64
    return z ^ (z >> 31)


def random_keys(seed: int, h: int, i: int, nb: int) -> np.ndarray:
    """Random selection keys of row (h, i): the top 24 bits of SplitMix64 at the counter
    seed + ((h * 4096 + i) * 4096 + j) for block j (exact integers, so the GPU's order,
    ties to the lower index, is the same)."""
    base = (seed + (h * 4096 + i) * 4096) & _MASK64
    return np.array([float(splitmix64((base + j) & _MASK64) >> 40) for j in range(nb)])


def select_row(P_i, vbar_i, Vb_h, WOh, n_cand: int, c: int, rounds: int, rho: float,
               h: int = 0, i: int = 0, variant: Variant = RESS) -> RowSelection:
    """Initial selection (Eq. 7) and R restoration rounds (Eq. 13-17) for one row."""
    nb = P_i.size
    _, _, r = residual_contributions(P_i, vbar_i, Vb_h, WOh)
    if variant.key == "drift":
        key = cut_keys(drift_scores(r), P_i)
    elif variant.key == "probability":
        key = np.array(P_i, dtype=np.float64)
    elif variant.key == "random":
        key = random_keys(variant.seed, h, i, nb)
    else:
        raise ValueError(variant.key)
    if variant.maximize == "full":  # keep the smallest keys: drop the largest drifts
        key = -key
    sign = -1.0 if variant.maximize in ("swap", "full") else 1.0  # restoration direction

    # initial selection: keep the c_h candidates with the largest key, drop the rest
    keep = top_m(key[:n_cand], c)
    D = np.zeros(nb, dtype=bool)
    D[:n_cand] = True
    D[keep] = False
    notes = [("cut", _gap(ranked(key[:n_cand]), c, 0.0))]
    if variant.cdf > 0:
        if rounds:
            raise ValueError("the CDF threshold is defined without restoration rounds")
        tau = variant.cdf
        mass = float(P_i[~D].sum())  # kept candidates and the always-kept blocks
        rest = np.nonzero(D[:n_cand])[0]
        order = rest[top_m(key[rest], rest.size)] if rest.size else rest
        masses = [mass]
        n_add = 0
        while n_add < order.size and mass < tau:
            mass += float(P_i[order[n_add]])
            masses.append(mass)
            n_add += 1
        D[order[:n_add]] = False
        keys_sorted = ranked(key[rest]) if rest.size else rest
        notes += [("cdf", x) for x in _cdf_margins(masses, tau, keys_sorted, n_add)]
    J, a, K = objective(D, P_i, r)
    res = RowSelection(h, i, False, D.copy(), D.copy(), J, J, [])
    for kind, value in notes:
        res.note(kind, value)
    for rnd, m_r in enumerate(swap_schedule(c, rounds, rho)):
        inD, gain_res, outD, gain_drop = round_gains(D, n_cand, P_i, r, J, a, K)
        m = min(m_r, inD.size, outD.size)
        if m == 0:
            res.J_trace.append(J)
            continue
        floor = 1e-30 * J
        gain_res, gain_drop = sign * gain_res, sign * gain_drop
        res.note("restore", _gap(ranked(gain_res), m, floor), rnd)
        res.note("drop", _gap(ranked(gain_drop), m, floor), rnd)
        restore = inD[top_m(gain_res, m)]
        drop = outD[top_m(gain_drop, m)]
        D[restore] = False
        D[drop] = True
        res.swaps += m
        J, a, K = objective(D, P_i, r)
        res.J_trace.append(J)
        res.note("track", _track_margin(J, res.J_best), rnd)
        if (J < res.J_best) if sign > 0 else (J > res.J_best):
            res.J_best = J
            res.D_best = D.copy()
    return res


def dense_row(h: int, i: int, nb: int) -> RowSelection:
    """Query blocks holding special tokens are not sparsified: everything kept, J = 0."""
    z = np.zeros(nb, dtype=bool)
    return RowSelection(h, i, True, z, z.copy(), 0.0, 0.0, [], math.inf)


@dataclass
class Pooled:
    """Block-pooled inputs of one layer: queries over query blocks of q_block tokens (64, or
    128 on the paper's own grid, Appendix F), keys and values over 64-token key blocks."""
    Qb: np.ndarray
    Kb: np.ndarray
    Vb: np.ndarray
    n_tokens: int
    n_special: int
    q_block: int = BLOCK

    @property
    def heads(self):
        return self.Qb.shape[0]

    @property
    def nb(self):
        """Key blocks."""
        return self.Kb.shape[1]

    @property
    def nq(self):
        """Query blocks (the rows of the selection)."""
        return self.Qb.shape[1]

    @property
    def n_cand(self):
        """Candidate key blocks |cal_P|."""
        return n_candidates(self.n_tokens, self.n_special)

    @property
    def n_qcand(self):
        """Query blocks made of patch tokens only: the sparsified rows."""
        return n_candidates(self.n_tokens, self.n_special, self.q_block)


def pool(Q, K, V, n_special: int, q_block: int = BLOCK) -> Pooled:
    return Pooled(pool_blocks(Q, q_block), pool_blocks(K), pool_blocks(V), Q.shape[0], n_special,
                  q_block)


def row_quantities(pooled: Pooled, h: int, i: int):
    """P_i and v_bar_i of one row."""
    P_i = pooled_attention_row(pooled.Qb[h, i], pooled.Kb[h])
    return P_i, dense_pooled_output(P_i, pooled.Vb[h])


def ress_select(pooled: Pooled, W_o, c_h, rounds: int, rho: float = 0.5, rows=None,
                variant: Variant = RESS):
    """ReSS selection (or one of its ablation variants) for every (h, i) row, or for the
    given list of rows.

    Returns {(h, i): RowSelection}.
    """
    H, nq, d_h = pooled.Qb.shape
    nb, n_cand = pooled.nb, pooled.n_cand
    if rows is None:
        rows = [(h, i) for h in range(H) for i in range(nq)]
    out = {}
    for h, i in rows:
        if i >= pooled.n_qcand:
            out[(h, i)] = dense_row(h, i, nb)
            continue
        P_i, vbar_i = row_quantities(pooled, h, i)
        out[(h, i)] = select_row(P_i, vbar_i, pooled.Vb[h], head_projection(W_o, h, d_h),
                                 n_cand, int(c_h[h]), rounds, rho, h, i, variant)
    return out


def drift_of(pooled: Pooled, W_o, h: int, i: int, D: np.ndarray) -> float:
    """J_i^h(D) of Eq. 12 for an arbitrary drop set D (bool over key blocks)."""
    d_h = pooled.Qb.shape[2]
    P_i, vbar_i = row_quantities(pooled, h, i)
    _, _, r = residual_contributions(P_i, vbar_i, pooled.Vb[h], head_projection(W_o, h, d_h))
    return objective(np.asarray(D, dtype=bool), P_i, r)[0]


# ----------------------------------------------------------------------------------------
# Sec. 3 step (3): exact attention over the kept blocks
# ----------------------------------------------------------------------------------------
def block_sparse_attention(Q, K, V, kept, rows, block: int = BLOCK, q_block: int = None) -> dict:
    """For every query token of query block i and head h: softmax(q k^T / sqrt(d_h)) over
    the tokens of the kept key blocks of (h, i), renormalised among them, times V.  Query
    blocks are q_block tokens (default: the key block size).

    kept: {(h, i): ascending key-block indices}.  Returns {(h, i): [rows_i, d_h] float64}.
    """
    N, H, d = Q.shape
    qb = block if q_block is None else q_block
    out = {}
    for h, i in rows:
        q = np.asarray(Q[i * qb: min(N, (i + 1) * qb), h], dtype=np.float64)
        idx = np.concatenate([np.arange(j * block, min(N, (j + 1) * block))
                              for j in kept[(h, i)]])
        k = np.asarray(K[idx, h], dtype=np.float64)
        v = np.asarray(V[idx, h], dtype=np.float64)
        s = (q @ k.T) / math.sqrt(d)
        p = np.exp(s - s.max(axis=1, keepdims=True))
        p /= p.sum(axis=1, keepdims=True)
        out[(h, i)] = p @ v
    return out


def csr_from_selection(sel: dict, H: int, nb: int):
    """Row-major (h, i) kept lists as CSR (row_ptr [H nb + 1], col_idx) in int32."""
    row_ptr = np.zeros(H * nb + 1, dtype=np.int64)
    cols = []
    for h in range(H):
        for i in range(nb):
            k = sel[(h, i)].kept()
            cols.append(k)
            row_ptr[h * nb + i + 1] = row_ptr[h * nb + i] + k.size
    return row_ptr.astype(np.int32), np.concatenate(cols).astype(np.int32)


# ----------------------------------------------------------------------------------------
# Sec. 3: what the attention sublayer adds to the residual stream
# ----------------------------------------------------------------------------------------
def residual_update(x, O, W_o):
    """x + O W_o^T: the pre-LN residual update x_{l+1} = x_l + f_l(x_l) of the attention
    sublayer (Sec. 3), with O [N, H d_h] the concatenated head outputs and W_o [d, H d_h] the
    output projection as a Linear weight (out x in).  x may be None (the update alone)."""
    y = np.asarray(O, dtype=np.float64) @ np.asarray(W_o, dtype=np.float64).T
    return y if x is None else np.asarray(x, dtype=np.float64) + y


def token_drift(O_a, O_b, W_o, block: int = BLOCK) -> np.ndarray:
    """Per query block: the squared Euclidean norm, over the block's query tokens and the
    residual dimension, of W_o (O_a - O_b), the change one attention output leaves in the
    residual stream relative to another (Sec. 3's token-level reference, with O_a the sparse
    and O_b the dense output).  Returns float64 [nb]."""
    delta = residual_update(None, np.asarray(O_a, np.float64) - np.asarray(O_b, np.float64), W_o)
    N = delta.shape[0]
    return np.array([float((delta[i * block: min(N, (i + 1) * block)] ** 2).sum())
                     for i in range(n_blocks(N, block))])
