"""Pins of the CPU oracle against what the paper and the mathematics fix (no GPU).

Each pin reaches the oracle's result by another route: PyTorch's scaled_dot_product_attention
and F.linear (library routines for softmax attention and the output projection), numpy's
reduceat (block sums), the paper's closed forms (Eq. 4, 9, 14-16), brute-force search over
every drop set, and invariants (scale, permutation, track-best, schedule totals).
"""
import itertools
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle as O
import synth

torch.set_default_dtype(torch.float64)


# ---------------------------------------------------------------------------------------
# small layers
# ---------------------------------------------------------------------------------------
def small_layer(n_tokens=778, n_special=10, heads=2, d_model=128, seed=1):
    d = synth.make_random_layer(n_tokens, heads, d_model, seed)
    X = {k: synth.bf16_to_f32(v).astype(np.float64) for k, v in d.items()}
    return X, n_special


def sdpa(q, k, v, mask=None):
    """Library softmax attention in float64: q [M, d], k/v [L, d], mask [M, L] bool."""
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a))[None, None]
    m = None if mask is None else torch.from_numpy(mask)[None, None]
    return F.scaled_dot_product_attention(t(q), t(k), t(v), attn_mask=m)[0, 0].numpy()


def pooled_output_via_library(pooled, h, i, D=None):
    """Renormalised pooled attention output of row (h, i) with the blocks of D masked."""
    q = pooled.Qb[h, i][None]
    mask = None if D is None else (~np.asarray(D, dtype=bool))[None]
    return sdpa(q, pooled.Kb[h], pooled.Vb[h], mask)[0]


def residual_drift_via_library(pooled, W_o, h, i, D):
    """||y_masked - y_dense||^2 with y = F.linear(concat_h pooled outputs, W_o): the change
    the masked attention sublayer leaves in the residual stream (Sec. 3, Eq. 11-12)."""
    H = pooled.heads
    dense = np.concatenate([pooled_output_via_library(pooled, g, i) for g in range(H)])
    masked = dense.copy()
    d_h = pooled.Qb.shape[2]
    masked[h * d_h:(h + 1) * d_h] = pooled_output_via_library(pooled, h, i, D)
    W = torch.from_numpy(W_o)
    y0 = F.linear(torch.from_numpy(dense), W)
    y1 = F.linear(torch.from_numpy(masked), W)
    return float(((y1 - y0) ** 2).sum())


@pytest.fixture(scope="module")
def layer():
    X, ns = small_layer()
    pooled = O.pool(X["Q"], X["K"], X["V"], ns)
    return X, pooled


# ---------------------------------------------------------------------------------------
# pooling and the pooled attention map
# ---------------------------------------------------------------------------------------
def test_shapes_of_the_block_grid():
    wl = synth.WORKLOADS["vggt_v32"]
    assert O.n_blocks(wl.n_tokens) == 687
    assert O.n_candidates(wl.n_tokens, wl.n_special) == 684
    wl1 = synth.WORKLOADS["tiny_v2"]
    assert (O.n_blocks(wl1.n_tokens), O.n_candidates(wl1.n_tokens, wl1.n_special)) == (43, 42)
    assert int(wl1.budgets()[0]) == 21 and int(wl.budgets()[0]) == 68


def test_pool_blocks_matches_reduceat(layer):
    X, pooled = layer
    N = X["Q"].shape[0]
    starts = np.arange(0, N, 64)
    counts = np.diff(np.append(starts, N))
    for name, got in (("Q", pooled.Qb), ("K", pooled.Kb), ("V", pooled.Vb)):
        ref = np.add.reduceat(X[name], starts, axis=0) / counts[:, None, None]
        np.testing.assert_allclose(got, np.transpose(ref, (1, 0, 2)), rtol=1e-13, atol=1e-13)
    assert counts[-1] == N - 64 * (len(starts) - 1) == 10   # ragged tail block


def test_dense_pooled_output_is_library_attention(layer):
    """Eq. 1 with P from the pooled softmax equals softmax attention at block level."""
    _, pooled = layer
    for h in range(pooled.heads):
        for i in (0, 5, pooled.nb - 1):
            P_i, vbar = O.row_quantities(pooled, h, i)
            assert abs(P_i.sum() - 1) < 1e-13 and (P_i > 0).all()
            np.testing.assert_allclose(vbar, pooled_output_via_library(pooled, h, i),
                                       rtol=1e-12, atol=1e-13)


def test_single_block_masking_identity(layer):
    """Eq. 3-4: masking block j gives v_bar + P/(1-P) (v_bar - V_j) exactly."""
    _, pooled = layer
    h, i = 1, 3
    P_i, vbar = O.row_quantities(pooled, h, i)
    for j in range(pooled.nb):
        D = np.zeros(pooled.nb, dtype=bool)
        D[j] = True
        direct = pooled_output_via_library(pooled, h, i, D)
        closed = vbar + P_i[j] / (1 - P_i[j]) * (vbar - pooled.Vb[h, j])
        np.testing.assert_allclose(direct, closed, rtol=1e-11, atol=1e-12)


# ---------------------------------------------------------------------------------------
# drift score and objective
# ---------------------------------------------------------------------------------------
def test_drift_score_equals_gram_expansion(layer):
    """Eq. 6 == Eq. 9: s_ij = P_ij sqrt(v^T M v - 2 v^T M V_j + V_j^T M V_j), M = W^T W."""
    X, pooled = layer
    d_h = 64
    for h in range(pooled.heads):
        WOh = O.head_projection(X["W_o"], h, d_h)
        M = WOh.T @ WOh                                              # Eq. 8
        P_i, vbar = O.row_quantities(pooled, h, 4)
        _, _, r = O.residual_contributions(P_i, vbar, pooled.Vb[h], WOh)
        s = O.drift_scores(r)
        Vb = pooled.Vb[h]
        q = vbar @ M @ vbar - 2 * (Vb @ M @ vbar) + np.einsum("jd,de,je->j", Vb, M, Vb)
        np.testing.assert_allclose(s, P_i * np.sqrt(np.maximum(q, 0)), rtol=1e-9)


def test_objective_equals_measured_residual_drift(layer):
    """Eq. 10-12: G/K^2 from the contribution vectors equals the change the masked
    attention output leaves after the output projection, for random drop sets."""
    X, pooled = layer
    rng = np.random.default_rng(0)
    for h in range(pooled.heads):
        for i in (0, 7, 11):
            for size in (1, 3, 6, 12):
                D = np.zeros(pooled.nb, dtype=bool)
                D[rng.choice(pooled.n_cand, size, replace=False)] = True
                J = O.drift_of(pooled, X["W_o"], h, i, D)
                ref = residual_drift_via_library(pooled, X["W_o"], h, i, D)
                assert J == pytest.approx(ref, rel=1e-9, abs=1e-18)


def test_single_drop_objective_is_squared_cut_key(layer):
    """Sec. 4.3: for D = {j}, Eq. 12 reduces to the square of the Eq. 7 key."""
    X, pooled = layer
    h, i = 0, 2
    P_i, vbar = O.row_quantities(pooled, h, i)
    _, _, r = O.residual_contributions(P_i, vbar, pooled.Vb[h], O.head_projection(X["W_o"], h, 64))
    key = O.cut_keys(O.drift_scores(r), P_i)
    for j in range(pooled.n_cand):
        D = np.zeros(pooled.nb, dtype=bool)
        D[j] = True
        assert O.objective(D, P_i, r)[0] == pytest.approx(key[j] ** 2, rel=1e-11)


def test_round_gains_match_closed_form(layer):
    """Eq. 14-16: the directly recomputed gains equal G/K^2 - (G + dG)/(K + u)^2 with
    dG = -/+ 2 d^T M g + s^2 computed from M_h = W_O^h^T W_O^h."""
    X, pooled = layer
    h, i = 1, 6
    WOh = O.head_projection(X["W_o"], h, 64)
    M = WOh.T @ WOh
    P_i, vbar = O.row_quantities(pooled, h, i)
    _, dvec, r = O.residual_contributions(P_i, vbar, pooled.Vb[h], WOh)
    s = O.drift_scores(r)
    D = np.zeros(pooled.nb, dtype=bool)
    D[[0, 2, 3, 7, 9, 10]] = True
    J, a, K = O.objective(D, P_i, r)
    g = dvec[D].sum(0)
    G = g @ M @ g
    assert J == pytest.approx(G / K ** 2, rel=1e-11)
    inD, gr, outD, gd = O.round_gains(D, pooled.n_cand, P_i, r, J, a, K)
    for k, gain in zip(inD, gr):
        dG = -2 * dvec[k] @ M @ g + s[k] ** 2                       # Eq. 14
        assert gain == pytest.approx(G / K ** 2 - (G + dG) / (K + P_i[k]) ** 2, rel=1e-8)
    for k, gain in zip(outD, gd):
        dG = 2 * dvec[k] @ M @ g + s[k] ** 2                        # Eq. 15
        assert gain == pytest.approx(G / K ** 2 - (G + dG) / (K - P_i[k]) ** 2, rel=1e-8)


# ---------------------------------------------------------------------------------------
# selection
# ---------------------------------------------------------------------------------------
def test_swap_schedule_totals():
    """Eq. 17: rho 2^-(r+1) c per round, at most rho (1 - 2^-R) c in total; paper default
    rho = 0.5, R = 5 gives 0.484 c."""
    assert O.swap_schedule(68, 3, 0.5) == [17, 8, 4]
    assert O.swap_schedule(214, 3, 0.5) == [53, 26, 13]
    assert O.swap_schedule(21, 2, 0.5) == [5, 2]
    for c in range(2, 400):
        for R in range(0, 8):
            assert sum(O.swap_schedule(c, R, 0.5)) <= 0.5 * (1 - 2.0 ** -R) * c + 1e-12
    assert 0.5 * (1 - 2 ** -5) == pytest.approx(0.484, abs=5e-4)


def test_initial_selection_single_drop_is_brute_force_optimum(layer):
    """|D| = 1: the Eq. 7 selection drops the block whose removal leaves the least drift,
    found by measuring every single-block removal through the library path."""
    X, pooled = layer
    c = pooled.n_cand - 1
    for h in range(pooled.heads):
        for i in (0, 4, 9):
            sel = O.ress_select(pooled, X["W_o"], [c] * pooled.heads, 0, rows=[(h, i)])[(h, i)]
            drifts = []
            for j in range(pooled.n_cand):
                D = np.zeros(pooled.nb, dtype=bool)
                D[j] = True
                drifts.append(residual_drift_via_library(pooled, X["W_o"], h, i, D))
            assert np.nonzero(sel.D0)[0].tolist() == [int(np.argmin(drifts))]


@pytest.mark.parametrize("c", [3, 6, 9])
def test_brute_force_bounds_restoration(layer, c):
    """Track-best restoration lands between the exhaustive optimum of Eq. 2 and the
    initial selection: J_opt <= J_ReSS <= J_0, and the returned set has the claimed J."""
    X, pooled = layer
    n = pooled.n_cand
    assert n == 12
    W = X["W_o"]
    for h in range(pooled.heads):
        for i in (1, 8):
            sel = O.ress_select(pooled, W, [c] * pooled.heads, 5, rows=[(h, i)])[(h, i)]
            P_i, vbar = O.row_quantities(pooled, h, i)
            _, _, r = O.residual_contributions(P_i, vbar, pooled.Vb[h], O.head_projection(W, h, 64))
            best = math.inf
            for comb in itertools.combinations(range(n), n - c):
                D = np.zeros(pooled.nb, dtype=bool)
                D[list(comb)] = True
                best = min(best, O.objective(D, P_i, r)[0])
            assert sel.D_best[:n].sum() == n - c and not sel.D_best[n:].any()
            assert best <= sel.J_best * (1 + 1e-12)
            assert sel.J_best <= sel.J0
            measured = residual_drift_via_library(pooled, W, h, i, sel.D_best)
            assert sel.J_best == pytest.approx(measured, rel=1e-9)


def test_track_best_and_monotone_in_rounds(layer):
    """J_best = min(J_0, J after each round) and, since m_r does not depend on R, one
    more round never raises J_best."""
    X, pooled = layer
    rows = [(h, i) for h in range(pooled.heads) for i in range(pooled.n_cand)]
    prev = None
    for R in range(0, 7):
        sel = O.ress_select(pooled, X["W_o"], [5] * pooled.heads, R, rows=rows)
        for key, s in sel.items():
            assert s.J_best == min([s.J0] + s.J_trace)
            assert len(s.J_trace) == R
            if prev is not None:
                assert s.J_best <= prev[key].J_best
                assert s.J_trace[:R - 1] == prev[key].J_trace
        prev = sel


def test_budget_is_preserved_and_special_blocks_kept(layer):
    X, pooled = layer
    sel = O.ress_select(pooled, X["W_o"], [4, 7], 3)
    for (h, i), s in sel.items():
        kept = s.kept()
        if i >= pooled.n_cand:
            assert s.dense and kept.tolist() == list(range(pooled.nb)) and s.J_best == 0
        else:
            assert int((kept < pooled.n_cand).sum()) == [4, 7][h]
            assert kept[-1] == pooled.nb - 1 and np.all(np.diff(kept) > 0)


def test_scale_invariance(layer):
    """W_o -> alpha W_o leaves every choice unchanged and scales J by alpha^2."""
    X, pooled = layer
    a = 3.0
    s1 = O.ress_select(pooled, X["W_o"], [5, 5], 3)
    s2 = O.ress_select(pooled, a * X["W_o"], [5, 5], 3)
    for k in s1:
        assert (s1[k].D_best == s2[k].D_best).all()
        assert s2[k].J_best == pytest.approx(a * a * s1[k].J_best, rel=1e-10, abs=1e-30)


def test_candidate_permutation_equivariance():
    """Permuting whole candidate key blocks (tokens of K and V) permutes the drop sets."""
    X, ns = small_layer(seed=3)
    pooled = O.pool(X["Q"], X["K"], X["V"], ns)
    perm = np.random.default_rng(5).permutation(pooled.n_cand)
    tok = np.arange(X["K"].shape[0])
    newtok = tok.copy()
    for dst, src in enumerate(perm):
        newtok[dst * 64:(dst + 1) * 64] = tok[src * 64:(src + 1) * 64]
    pooled2 = O.pool(X["Q"], X["K"][newtok], X["V"][newtok], ns)
    rows = [(h, i) for h in range(2) for i in range(0, 12, 3)]
    s1 = O.ress_select(pooled, X["W_o"], [5, 5], 3, rows=rows)
    s2 = O.ress_select(pooled2, X["W_o"], [5, 5], 3, rows=rows)
    for k in rows:
        assert (s2[k].D_best[:12] == s1[k].D_best[:12][perm]).all()
        assert s2[k].J_best == pytest.approx(s1[k].J_best, rel=1e-9)


def test_deterministic(layer):
    X, pooled = layer
    a = O.ress_select(pooled, X["W_o"], [6, 6], 4)
    b = O.ress_select(pooled, X["W_o"], [6, 6], 4)
    for k in a:
        assert (a[k].D_best == b[k].D_best).all() and a[k].J_best == b[k].J_best


# ---------------------------------------------------------------------------------------
# token-level attention
# ---------------------------------------------------------------------------------------
def _token_mask(kept, N, H, nb):
    mask = np.zeros((H, N, N), dtype=bool)
    for (h, i), cols in kept.items():
        for j in cols:
            mask[h, i * 64:min(N, i * 64 + 64), j * 64:min(N, j * 64 + 64)] = True
    return mask


def test_zero_sparsity_is_dense_attention(layer):
    """c_h = |P| keeps every block; the output equals library dense attention."""
    X, pooled = layer
    sel = O.ress_select(pooled, X["W_o"], [pooled.n_cand] * 2, 3)
    kept = {k: s.kept() for k, s in sel.items()}
    assert all(len(v) == pooled.nb for v in kept.values())
    out = O.block_sparse_attention(X["Q"], X["K"], X["V"], kept, list(kept))
    N = X["Q"].shape[0]
    for h in range(2):
        ref = sdpa(X["Q"][:, h], X["K"][:, h], X["V"][:, h])
        for i in range(pooled.nb):
            np.testing.assert_allclose(out[(h, i)], ref[i * 64:min(N, i * 64 + 64)],
                                       rtol=1e-10, atol=1e-12)


def test_block_sparse_attention_is_masked_library_attention(layer):
    """Sec. 3 step (3): exact attention over the kept blocks, renormalised among them,
    equals library attention with the dropped blocks masked out."""
    X, pooled = layer
    sel = O.ress_select(pooled, X["W_o"], [3, 8], 2)
    kept = {k: s.kept() for k, s in sel.items()}
    out = O.block_sparse_attention(X["Q"], X["K"], X["V"], kept, list(kept))
    N = X["Q"].shape[0]
    mask = _token_mask(kept, N, 2, pooled.nb)
    for h in range(2):
        ref = sdpa(X["Q"][:, h], X["K"][:, h], X["V"][:, h], mask[h])
        for i in range(pooled.nb):
            np.testing.assert_allclose(out[(h, i)], ref[i * 64:min(N, i * 64 + 64)],
                                       rtol=1e-10, atol=1e-12)


def test_csr_layout(layer):
    X, pooled = layer
    sel = O.ress_select(pooled, X["W_o"], [3, 8], 2)
    rp, ci = O.csr_from_selection(sel, 2, pooled.nb)
    assert rp[0] == 0 and rp[-1] == ci.size
    ns = pooled.nb - pooled.n_cand
    lens = np.diff(rp).reshape(2, pooled.nb)
    assert (lens[0, :pooled.n_cand] == 3 + ns).all() and (lens[1, :pooled.n_cand] == 8 + ns).all()
    assert (lens[:, pooled.n_cand:] == pooled.nb).all()


# ---------------------------------------------------------------------------------------
# Sec. 3: residual update and token-level drift
# ---------------------------------------------------------------------------------------
def test_residual_update_elementwise_by_loops():
    """y[t, o] = x[t, o] + sum_k O[t, k] W_o[o, k], written out with loops on a small case
    whose W_o is not symmetric (a transposed operand fails it)."""
    rng = np.random.default_rng(7)
    N, d = 5, 6
    x, Ob, W = rng.normal(size=(N, d)), rng.normal(size=(N, d)), rng.normal(size=(d, d))
    y = O.residual_update(x, Ob, W)
    for t in range(N):
        for o in range(d):
            acc = x[t, o]
            for k in range(d):
                acc += Ob[t, k] * W[o, k]
            assert y[t, o] == pytest.approx(acc, rel=1e-13, abs=1e-13)
    assert np.allclose(O.residual_update(None, Ob, W), y - x, rtol=0, atol=1e-13)


def test_residual_update_is_the_output_projection_linear():
    """The update equals F.linear with W_o as the Linear weight (out x in), and with an
    identity W_o it is x + O."""
    rng = np.random.default_rng(8)
    x, Ob = rng.normal(size=(9, 16)), rng.normal(size=(9, 16))
    W = rng.normal(size=(16, 16))
    ref = torch.from_numpy(x) + F.linear(torch.from_numpy(Ob), torch.from_numpy(W))
    assert np.allclose(O.residual_update(x, Ob, W), ref.numpy(), rtol=1e-12, atol=1e-12)
    assert np.allclose(O.residual_update(x, Ob, np.eye(16)), x + Ob, rtol=0, atol=1e-14)


def test_token_drift_definition_and_invariants(layer):
    """Token drift per block: zero for identical outputs, the squared norm of the difference
    of the two residual updates, scaling by alpha^2 with W_o, blocks summing to the whole."""
    rng = np.random.default_rng(9)
    N, d = 200, 32
    Oa, Ob, W = rng.normal(size=(N, d)), rng.normal(size=(N, d)), rng.normal(size=(d, d))
    dr = O.token_drift(Oa, Ob, W, block=64)
    assert dr.shape == (4,)
    assert np.all(O.token_drift(Oa, Oa, W, block=64) == 0)
    ya, yb = O.residual_update(None, Oa, W), O.residual_update(None, Ob, W)
    for b in range(4):
        sl = slice(64 * b, min(N, 64 * (b + 1)))
        assert dr[b] == pytest.approx(float(np.linalg.norm(ya[sl] - yb[sl]) ** 2), rel=1e-12)
    assert np.allclose(O.token_drift(Oa, Ob, 3.0 * W, block=64), 9.0 * dr, rtol=1e-12)
    assert dr.sum() == pytest.approx(float(((ya - yb) ** 2).sum()), rel=1e-12)


# ---------------------------------------------------------------------------------------
# Ablation variants (Sec. 6): probability keys, random keys, maximised drift
# ---------------------------------------------------------------------------------------
def test_splitmix64_reference_outputs():
    """The counter-based generator behind the random variant reproduces SplitMix64's
    published outputs for seed 0 (tests/golden/splitmix64_seed0.txt)."""
    import pathlib
    path = pathlib.Path(__file__).with_name("golden") / "splitmix64_seed0.txt"
    want = [int(l, 16) for l in path.read_text().splitlines() if l.startswith("0x")]
    state, got = 0, []
    for _ in want:
        got.append(O.splitmix64(state))
        state = (state + 0x9E3779B97F4A7C15) & ((1 << 64) - 1)
    assert got == want


def _variant_rows(layer, variant, rounds=3):
    X, pooled = layer
    H, nb = pooled.heads, pooled.nb
    c = [max(2, pooled.n_cand // 4)] * H
    rows = [(h, i) for h in range(H) for i in range(0, pooled.n_cand, 3)]
    return pooled, c, O.ress_select(pooled, X["W_o"], c, rounds, 0.5, rows=rows, variant=variant)


def test_probability_variant_is_top_k_by_pooled_mass(layer):
    """key = P_ij with no rounds keeps exactly the c_h candidates of largest pooled
    probability (ties to the lower index), found here by a stable argsort."""
    pooled, c, sel = _variant_rows(layer, O.Variant(key="probability"), rounds=0)
    for (h, i), s in sel.items():
        P_i, _ = O.row_quantities(pooled, h, i)
        order = np.argsort(-P_i[:pooled.n_cand], kind="stable")[:c[h]]
        assert set(np.nonzero(~s.D_best[:pooled.n_cand])[0]) == set(order)


def test_random_variant_keys(layer):
    """Random keys: the same seed gives the same sets, another seed other sets, and every
    row keeps exactly c_h candidates."""
    pooled, c, a = _variant_rows(layer, O.Variant(key="random", seed=5), rounds=0)
    _, _, b = _variant_rows(layer, O.Variant(key="random", seed=5), rounds=0)
    _, _, o = _variant_rows(layer, O.Variant(key="random", seed=6), rounds=0)
    assert all(np.array_equal(a[k].D_best, b[k].D_best) for k in a)
    assert any(not np.array_equal(a[k].D_best, o[k].D_best) for k in a)
    for (h, i), s in a.items():
        assert (~s.D_best).sum() == c[h] + (pooled.nb - pooled.n_cand)


def test_maximised_drift_variants(layer):
    """Flipping the sign (Fig. 8): "swap" keeps ReSS's initial set and its rounds never
    lower the best J below J0; "full" keeps the smallest Eq. 7 keys; the best J is the
    largest J seen, and it does not decrease with more rounds."""
    pooled, c, ress = _variant_rows(layer, O.RESS)
    _, _, swap = _variant_rows(layer, O.Variant(maximize="swap"))
    _, _, full = _variant_rows(layer, O.Variant(maximize="full"))
    _, _, full2 = _variant_rows(layer, O.Variant(maximize="full"), rounds=2)
    for k in ress:
        assert np.array_equal(swap[k].D0, ress[k].D0)
        for v in (swap[k], full[k]):
            assert v.J_best >= v.J0
            assert v.J_best == max([v.J0] + v.J_trace)
        assert full[k].J_best >= full2[k].J_best
        h, i = k
        P_i, vbar_i = O.row_quantities(pooled, h, i)
        _, _, r = O.residual_contributions(P_i, vbar_i, pooled.Vb[h],
                                           O.head_projection(layer[0]["W_o"], h, 64))
        key = O.cut_keys(O.drift_scores(r), P_i)[:pooled.n_cand]
        smallest = set(np.argsort(key, kind="stable")[:c[h]])
        assert set(np.nonzero(~full[k].D0[:pooled.n_cand])[0]) == smallest


def test_cdf_threshold_probability_key_is_top_p(layer):
    """CDF threshold on the probability key (Table 3's "+ CDF threshold" row): the kept
    candidates are the first n of a stable descending argsort of P, n the larger of c_h and
    the shortest prefix whose mass, with the always-kept blocks, reaches tau (np.cumsum)."""
    for tau in (0.3, 0.6, 0.9, 0.99):
        pooled, c, sel = _variant_rows(layer, O.Variant(key="probability", cdf=tau), rounds=0)
        nc = pooled.n_cand
        for (h, i), s in sel.items():
            P_i, _ = O.row_quantities(pooled, h, i)
            order = np.argsort(-P_i[:nc], kind="stable")
            reach = P_i[nc:].sum() + np.cumsum(P_i[order])
            n_tau = int(np.searchsorted(reach >= tau, True)) + 1 if reach[-1] >= tau else nc
            n = max(c[h], n_tau)
            assert set(np.nonzero(~s.D_best[:nc])[0]) == set(order[:n]), (tau, h, i)


def test_cdf_threshold_invariants(layer):
    """With the drift key: a threshold at or below the mass of the top-c_h set changes
    nothing; otherwise the kept set contains ReSS's initial set, its mass reaches tau, and
    taking back its lowest-key added block falls below tau (the prefix is the shortest)."""
    pooled, c, base = _variant_rows(layer, O.RESS, rounds=0)
    _, _, low = _variant_rows(layer, O.Variant(cdf=1e-9), rounds=0)
    assert all(np.array_equal(low[k].D_best, base[k].D_best) for k in base)
    X = layer[0]
    for tau in (0.5, 0.8, 0.95):
        _, _, sel = _variant_rows(layer, O.Variant(cdf=tau), rounds=0)
        for (h, i), s in sel.items():
            P_i, vbar_i = O.row_quantities(pooled, h, i)
            kept = ~s.D_best
            assert (~base[(h, i)].D_best <= kept).all()
            added = np.nonzero(kept & base[(h, i)].D_best)[0]
            mass = P_i[kept].sum()
            if added.size == 0:
                assert P_i[~base[(h, i)].D_best].sum() >= tau or kept.all()
                continue
            _, _, r = O.residual_contributions(P_i, vbar_i, pooled.Vb[h],
                                               O.head_projection(X["W_o"], h, 64))
            key = O.cut_keys(O.drift_scores(r), P_i)
            last = added[np.lexsort((-added, key[added]))[0]]  # lowest key, highest index
            assert mass >= tau - 1e-12 or kept[:pooled.n_cand].all()
            assert mass - P_i[last] < tau
            # every added block outranks every candidate still dropped
            still = np.nonzero(s.D_best[:pooled.n_cand])[0]
            if still.size:
                assert key[added].min() >= key[still].max()
    with pytest.raises(ValueError):
        _variant_rows(layer, O.Variant(cdf=0.9), rounds=1)


# ---------------------------------------------------------------------------------------
# The paper's grid (Appendix F): 128-token query blocks over 64-token key blocks
# ---------------------------------------------------------------------------------------
def test_query_block_128_pooling_is_the_weighted_pair_mean(layer):
    """A 128-token query block's mean is the token-count-weighted mean of its two 64-token
    halves (the ragged tail included)."""
    X, _ = layer
    Q = X["Q"]
    N = Q.shape[0]
    q64 = O.pool_blocks(Q, 64)
    q128 = O.pool_blocks(Q, 128)
    for i in range(q128.shape[1]):
        n0 = min(64, N - 128 * i)
        n1 = max(0, min(64, N - 128 * i - 64))
        want = (n0 * q64[:, 2 * i] + (n1 * q64[:, 2 * i + 1] if n1 else 0.0)) / (n0 + n1)
        assert np.allclose(q128[:, i], want, rtol=1e-12, atol=1e-12)


def test_query_block_128_attention_is_two_64_blocks_with_the_same_list(layer):
    """Attention of a 128-token query block over a kept list equals that of its two 64-token
    halves over the same list (each query token attends the same keys)."""
    X, _ = layer
    nb = O.n_blocks(X["Q"].shape[0])
    rng = np.random.default_rng(3)
    kept = {(0, i): np.sort(rng.choice(nb, 5, replace=False)) for i in range(3)}
    a128 = O.block_sparse_attention(X["Q"], X["K"], X["V"], kept, list(kept), q_block=128)
    kept64 = {(0, 2 * i + s): kept[(0, i)] for i in range(3) for s in range(2)}
    a64 = O.block_sparse_attention(X["Q"], X["K"], X["V"], kept64, list(kept64))
    for i in range(3):
        assert np.allclose(a128[(0, i)], np.vstack([a64[(0, 2 * i)], a64[(0, 2 * i + 1)]]),
                           rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------------------------------
# Decision margins (which rows the GPU comparison excuses from the bit-exact rule)
# ---------------------------------------------------------------------------------------
def line_row(x):
    """A row whose drift lives on one residual axis, so every key and gain has a closed form.

    P is uniform (1/n over n candidate blocks, none always kept), W_O^h = I_64 and the pooled
    values are V_j = x_j e_0 with sum x_j = 0, so v_bar = 0 and e_j = -x_j e_0.  Then
    (Eq. 5-7, 10-12) the cut key of block j is |x_j| / (n - 1), and a drop set D has
    J(D) = (sum_{j in D} x_j)^2 / (n - |D|)^2; restoring k gives (S - x_k)^2 / (n - |D| + 1)^2
    and dropping k gives (S + x_k)^2 / (n - |D| - 1)^2 (Eq. 13-16).  The expected margins
    below were worked out by hand from these closed forms."""
    x = np.asarray(x, dtype=np.float64)
    n = x.size
    P = np.full(n, 1.0 / n)
    Vb = np.zeros((n, 64))
    Vb[:, 0] = x
    return P, P @ Vb, Vb, np.eye(64)


def _margins(sel):
    return [(m[0], m[-1]) if len(m) == 2 else (m[0], m[1], m[2]) for m in sel.margins]


def _assert_margins(sel, want):
    got = _margins(sel)
    assert [g[:-1] for g in got] == [w[:-1] for w in want], got
    for g, w in zip(got, want):
        assert g[-1] == pytest.approx(w[-1], rel=1e-12, abs=0), (g, w)
    assert sel.margin == pytest.approx(min(w[-1] for w in want), rel=1e-12)


def test_margin_of_the_eq7_cut(layer=None):
    """Keys |x_j| / 7 ranked 5, 4, 3.5 | 3, 2, 1.5, 1, 1 (over 7): keeping c = 3 decides
    between 3.5 and 3, a gap of 0.5 relative to 3.5."""
    sel = O.select_row(*line_row([5, -4, 3.5, -3, 2, -1.5, -1, -1]), 8, 3, 0, 0.5)
    _assert_margins(sel, [("cut", 1 / 7)])
    assert not sel.near_threshold


def test_margins_of_a_restoration_round(layer=None):
    """c = 3, rho = 1.5, one round of m = 2.  D0 = {3,...,7}, S = -4.5, J0 = 2.25.
    Restore gains 2.25 - (S - x_k)^2 / 16: 135/64 (k=3), 27/16 (k=5), 95/64 (k=6, 7),
    -25/64 (k=4); the cut between the 2nd and 3rd is (27/16 - 95/64) / (27/16) = 13/108.
    Drop gains 2.25 - (S + x_k)^2 / 4: 35/16 (k=0), 2 (k=2), -253/16 (k=1); the cut
    (2 + 253/16) / (253/16) = 285/253.  The new set {0, 2, 4, 6, 7} has J = 8.5^2 / 9, above
    J0: track-best margin (72.25/9 - 2.25) / 2.25 = 208/81, and the best set stays D0."""
    sel = O.select_row(*line_row([5, -4, 3.5, -3, 2, -1.5, -1, -1]), 8, 3, 1, 1.5)
    _assert_margins(sel, [("cut", 1 / 7), ("restore", 0, 13 / 108), ("drop", 0, 285 / 253),
                          ("track", 0, 208 / 81)])
    assert np.nonzero(sel.D_best)[0].tolist() == [3, 4, 5, 6, 7]
    assert sel.J_trace == [pytest.approx(72.25 / 9, rel=1e-14)]


def test_margins_of_track_best_comparisons(layer=None):
    """Keys over 7: 19, 9, 8 | 7, 6, 4, 2, 1 (cut 1/8).  rho = 2: round 0 swaps m = 3 (every
    kept candidate leaves, so the drop side has no cut: inf) and lowers J from 36 to 289/9:
    track margin (36 - 289/9) / 36 = 35/324, taken relative to the best so far (J0).  Round 1
    (m = 1) reaches J = 9: track margin (289/9 - 9) / (289/9) = 208/289, relative to the
    updated best 289/9.  The restore cuts are 3/19 and 693/4588, the round-1 drop cut 189/256;
    the row's margin is the round-0 track-best comparison."""
    sel = O.select_row(*line_row([6, -8, -1, 7, 9, 4, 2, -19]), 8, 3, 2, 2.0)
    _assert_margins(sel, [("cut", 1 / 8), ("restore", 0, 3 / 19), ("drop", 0, math.inf),
                          ("track", 0, 35 / 324), ("restore", 1, 693 / 4588),
                          ("drop", 1, 189 / 256), ("track", 1, 208 / 289)])
    assert sel.J0 == pytest.approx(36.0, rel=1e-14)
    assert sel.J_best == pytest.approx(9.0, rel=1e-14)


def test_margins_of_the_cdf_threshold(layer=None):
    """Probability key on P = (5, 3, 2, 1.5, 1, 0.5 | 3) / 16 (six candidates, one always-kept
    block), c = 1, tau = 0.75: the kept mass starts at 8/16 and grows to 11/16, then 13/16,
    so two blocks join (n_add = 2).  Margins: the Eq. 7 cut (5 - 3)/5 = 0.4; each running
    mass against tau, |8/16 - 3/4| / (3/4) = 1/3, then 1/12 and 1/12; the key gaps of the
    remaining candidates (3, 2, 1.5, 1, 0.5)/16 on both sides of the last joiner,
    (2 - 1.5)/2 = 1/4 and (3 - 2)/3 = 1/3."""
    P = np.array([5, 3, 2, 1.5, 1, 0.5, 3]) / 16.0
    Vb = np.random.default_rng(0).normal(size=(7, 64))
    sel = O.select_row(P, P @ Vb, Vb, np.eye(64), 6, 1, 0, 0.5,
                       variant=O.Variant(key="probability", cdf=0.75))
    _assert_margins(sel, [("cut", 0.4), ("cdf", 1 / 3), ("cdf", 1 / 12), ("cdf", 1 / 12),
                          ("cdf", 0.25), ("cdf", 1 / 3)])
    assert np.nonzero(~sel.D_best)[0].tolist() == [0, 1, 2, 6]


def test_margin_is_smallest_recorded_and_near_rule(layer):
    """On real rows the row margin is the smallest recorded decision margin, every round that
    swaps records one restore cut, one drop cut and one track-best comparison, and a row with
    equal keys at the Eq. 7 cut has margin 0 and is near-threshold."""
    X, pooled = layer
    sel = O.ress_select(pooled, X["W_o"], [4, 6], 3)
    for (h, i), s in sel.items():
        if s.dense:
            assert s.margins == [] and s.margin == math.inf
            continue
        assert s.margin == min(m[-1] for m in s.margins)
        assert s.margins[0][0] == "cut"
        swapping = [r for r, m in enumerate(O.swap_schedule([4, 6][h], 3, 0.5)) if m > 0]
        for kind in ("restore", "drop", "track"):
            assert [m[1] for m in s.margins if m[0] == kind] == swapping
    tie = O.select_row(*line_row([3, -3, 2, -2, 1, -1]), 6, 3, 0, 0.5)
    assert tie.margin == 0.0 and tie.near_threshold
