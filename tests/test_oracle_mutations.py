"""The pins must catch plausible mistakes: each case below plants one in the oracle (on the
CPU, through monkeypatch) and checks that at least one pin of test_oracle_pins fails."""
import math

import numpy as np
import pytest

import oracle as O
import oracle.ress_oracle as R
import test_oracle_pins as pins


def _fresh_layer():
    X, ns = pins.small_layer()
    return X, O.pool(X["Q"], X["K"], X["V"], ns)


PIN_SET = [
    pins.test_pool_blocks_matches_reduceat,
    pins.test_dense_pooled_output_is_library_attention,
    pins.test_single_block_masking_identity,
    pins.test_drift_score_equals_gram_expansion,
    pins.test_objective_equals_measured_residual_drift,
    pins.test_single_drop_objective_is_squared_cut_key,
    pins.test_round_gains_match_closed_form,
    pins.test_initial_selection_single_drop_is_brute_force_optimum,
    lambda layer: pins.test_brute_force_bounds_restoration(layer, 6),
    pins.test_budget_is_preserved_and_special_blocks_kept,
    pins.test_block_sparse_attention_is_masked_library_attention,
    lambda layer: pins.test_swap_schedule_totals(),
    pins.test_margin_of_the_eq7_cut,
    pins.test_margins_of_a_restoration_round,
    pins.test_margins_of_track_best_comparisons,
    pins.test_margins_of_the_cdf_threshold,
]


def _mut_pool_divides_by_block(X, block=R.BLOCK):
    N, H, d = X.shape
    out = np.empty((H, R.n_blocks(N, block), d))
    for j in range(out.shape[1]):
        out[:, j] = np.asarray(X[j * block:(j + 1) * block], dtype=np.float64).sum(0) / block
    return out


def _mut_softmax_scale(qbar_i, Kb_h):
    logits = Kb_h @ qbar_i / qbar_i.shape[-1]
    z = np.exp(logits - logits.max())
    return z / z.sum()


def _mut_head_rows(W_o, h, d_h):
    return np.asarray(W_o[h * d_h:(h + 1) * d_h, :], dtype=np.float64).T


def _mut_no_renorm(s, P_i):
    return s


def _mut_objective_K(D, P_i, r):
    a = r[D].sum(axis=0) if D.any() else np.zeros(r.shape[1])
    K = P_i[D].sum()
    return float(a @ a) / max(K, R.EPS) ** 2, a, K


def _mut_gain_sign(D, n_cand, P_i, r, J, a, K):
    inD = np.nonzero(D[:n_cand])[0]
    outD = np.nonzero(~D[:n_cand])[0]
    J_res = ((a[None] - r[inD]) ** 2).sum(1) / np.maximum(K + P_i[inD], R.EPS) ** 2
    J_drop = ((a[None] - r[outD]) ** 2).sum(1) / np.maximum(K - P_i[outD], R.EPS) ** 2
    return inD, J - J_res, outD, J - J_drop


def _mut_gain_K(D, n_cand, P_i, r, J, a, K):
    inD = np.nonzero(D[:n_cand])[0]
    outD = np.nonzero(~D[:n_cand])[0]
    J_res = ((a[None] - r[inD]) ** 2).sum(1) / max(K, R.EPS) ** 2
    J_drop = ((a[None] + r[outD]) ** 2).sum(1) / max(K, R.EPS) ** 2
    return inD, J - J_res, outD, J - J_drop


def _mut_dev_sign(P_i, vbar_i, Vb_h, WOh):
    e = Vb_h + vbar_i[None, :]
    dvec = P_i[:, None] * e
    return e, dvec, dvec @ WOh.T


def _mut_schedule_ceil(c, rounds, rho):
    return [int(math.ceil(rho * c / 2 ** (r + 1))) for r in range(rounds)]


def _mut_topm_smallest(values, m):
    order = sorted(range(values.size), key=lambda k: (values[k], k))
    return np.array(order[:m], dtype=np.int64)


def _mut_attention_scale(Q, K, V, kept, rows, block=R.BLOCK):
    out = {}
    N = Q.shape[0]
    for h, i in rows:
        q = np.asarray(Q[i * block:min(N, (i + 1) * block), h], dtype=np.float64)
        idx = np.concatenate([np.arange(j * block, min(N, (j + 1) * block)) for j in kept[(h, i)]])
        s = q @ np.asarray(K[idx, h]).T / Q.shape[2]
        p = np.exp(s - s.max(1, keepdims=True))
        out[(h, i)] = (p / p.sum(1, keepdims=True)) @ np.asarray(V[idx, h])
    return out


def _mut_gap_off_by_one(vals_sorted, m, floor):
    if m <= 0 or m + 1 >= vals_sorted.size:
        return math.inf
    a, b = vals_sorted[m], vals_sorted[m + 1]
    scale = max(abs(a), abs(b), floor)
    return (a - b) / scale if scale > 0 else 0.0


def _mut_gap_scale_next(vals_sorted, m, floor):
    if m <= 0 or m >= vals_sorted.size:
        return math.inf
    a, b = vals_sorted[m - 1], vals_sorted[m]
    scale = max(abs(b), floor)
    return (a - b) / scale if scale > 0 else 0.0


def _mut_track_over_new_J(J, J_best):
    return abs(J - J_best) / J if J > 0 else math.inf


def _mut_cdf_no_start_mass(masses, tau, keys_sorted, n_add):
    out = [abs(x - tau) / tau for x in masses[1:]]
    if keys_sorted.size:
        out += [R._gap(keys_sorted, n_add, 0.0), R._gap(keys_sorted, n_add - 1, 0.0)]
    return out


def _mut_cdf_one_side(masses, tau, keys_sorted, n_add):
    out = [abs(x - tau) / tau for x in masses]
    if keys_sorted.size:
        out += [R._gap(keys_sorted, n_add, 0.0)]
    return out


MUTATIONS = {
    "pool divides the ragged tail by 64": ("pool_blocks", _mut_pool_divides_by_block),
    "pooled logits scaled by 1/d": ("pooled_attention_row", _mut_softmax_scale),
    "W_O^h taken from rows": ("head_projection", _mut_head_rows),
    "Eq. 7 without the renormalisation factor": ("cut_keys", _mut_no_renorm),
    "K = dropped mass instead of remaining mass": ("objective", _mut_objective_K),
    "drop gain with the restore sign": ("round_gains", _mut_gain_sign),
    "gains ignore the change of K": ("round_gains", _mut_gain_K),
    "deviation v_bar + V_j": ("residual_contributions", _mut_dev_sign),
    "schedule rounded up": ("swap_schedule", _mut_schedule_ceil),
    "top-m takes the smallest": ("top_m", _mut_topm_smallest),
    "token attention scaled by 1/d": ("block_sparse_attention", _mut_attention_scale),
    "margin between the (m+1)-th and (m+2)-th": ("_gap", _mut_gap_off_by_one),
    "margin relative to the (m+1)-th value": ("_gap", _mut_gap_scale_next),
    "track-best margin relative to the new J": ("_track_margin", _mut_track_over_new_J),
    "CDF margins without the starting mass": ("_cdf_margins", _mut_cdf_no_start_mass),
    "CDF key gap on one side only": ("_cdf_margins", _mut_cdf_one_side),
}


@pytest.mark.parametrize("name", list(MUTATIONS))
def test_planted_mistake_is_caught(name, monkeypatch):
    attr, fn = MUTATIONS[name]
    monkeypatch.setattr(R, attr, fn)
    monkeypatch.setattr(O, attr, fn, raising=False)
    failures = 0
    for pin in PIN_SET:
        try:
            pin(_fresh_layer())
        except AssertionError:
            failures += 1
    assert failures > 0, f"no pin caught: {name}"


def test_unmutated_oracle_passes_every_pin():
    for pin in PIN_SET:
        pin(_fresh_layer())
