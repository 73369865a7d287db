"""GPU parity of every stage of the hot path against the CPU oracle (needs a GB300)."""
import numpy as np
import pytest

import oracle as O
import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():  # collected on CPU machines only to be deselected
    pytest.skip("no CUDA device", allow_module_level=True)

import gpu_harness as G  # noqa: E402


def layer_for(name, **kw):
    wl = synth.WORKLOADS[name].with_(**kw) if kw else synth.WORKLOADS[name]
    return G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), wl.rounds, wl.rho), wl


@pytest.fixture(scope="module")
def tiny():
    layer, _ = layer_for("tiny_v2")
    return layer.run()


@pytest.fixture(scope="module")
def v8():
    layer, _ = layer_for("vggt_v8")
    return layer.run()


def test_prepare_wo_factor(tiny):
    F = tiny.buf.F.cpu().numpy().astype(np.float64)
    W = tiny.W_o()
    for h in range(tiny.H):
        Wh = O.head_projection(W, h, 64)
        M = Wh.T @ Wh
        np.testing.assert_allclose(F[h].T @ F[h], M, rtol=2e-5, atol=2e-6 * np.abs(M).max())
        assert np.allclose(np.tril(F[h], -1), 0)


def test_pooling(tiny):
    p = tiny.pooled()
    H, nb = tiny.H, tiny.nb
    for name, ref in (("qbar", p.Qb), ("kbar", p.Kb), ("vbar", p.Vb)):
        got = tiny.ws(name, shape=(H, nb, 64))
        np.testing.assert_allclose(got, ref, rtol=1e-5, atol=1e-6)


def test_pooled_map_and_scores(tiny):
    p = tiny.pooled()
    L = tiny.buf.layout
    P = tiny.ws("P", shape=(tiny.H, tiny.nb, L.ld))
    q = tiny.ws("q", shape=(tiny.H, tiny.nb, L.ld))
    W = tiny.W_o()
    for h in range(tiny.H):
        for i in range(0, tiny.ncand, 5):
            P_i, vbar = O.row_quantities(p, h, i)
            np.testing.assert_allclose(P[h, i, :tiny.nb], P_i, rtol=2e-5, atol=1e-9)
            e, _, _ = O.residual_contributions(P_i, vbar, p.Vb[h], O.head_projection(W, h, 64))
            Wh = O.head_projection(W, h, 64)
            q_ref = ((e @ Wh.T) ** 2).sum(1)
            np.testing.assert_allclose(q[h, i, :tiny.nb], q_ref, rtol=5e-4, atol=1e-6 * q_ref.max())


def test_initial_objective(tiny):
    """J of the initial selection (Eq. 7 then Eq. 12) on rows decided away from any tie."""
    sel = tiny.oracle_select()
    J0 = tiny.ws("J0", shape=(tiny.H, tiny.nb))
    D = tiny.drop_sets()
    checked = 0
    for (h, i), s in sel.items():
        if s.dense or s.near_threshold or not (D[h, i] == s.D_best).all():
            continue
        assert J0[h, i] == pytest.approx(s.J0, rel=G.DRIFT_REL)
        checked += 1
    assert checked > 0


@pytest.mark.parametrize("fixture", ["tiny", "v8"])
def test_drop_sets_and_drift(fixture, request):
    layer = request.getfixturevalue(fixture)
    sel = layer.oracle_select()
    r = G.compare_selection(layer, sel)
    G.check_selection(r)
    print(fixture, r)
    assert r["mismatched"] == 0, r
    assert r["exact"] >= 0.95 * (r["exact"] + r["near"])
    assert r["worst_row_rel"] <= G.DRIFT_REL
    assert r["sum_rel_gpu_vs_ref"] <= G.DRIFT_REL
    assert r["sum_rel_gpu_vs_oracle"] <= G.DRIFT_REL


@pytest.mark.parametrize("fixture", ["tiny", "v8"])
def test_csr_structure(fixture, request):
    layer = request.getfixturevalue(fixture)
    rp, ci = layer.csr()
    nb, nc = layer.nb, layer.ncand
    D = layer.drop_sets()
    assert rp[0] == 0 and rp[-1] == ci.size
    for h in range(layer.H):
        for i in range(nb):
            k = ci[rp[h * nb + i]:rp[h * nb + i + 1]]
            assert np.all(np.diff(k) > 0)
            if i >= nc:
                assert k.tolist() == list(range(nb))
            else:
                assert k.size == layer.c_h[h] + nb - nc
                assert np.array_equal(k, np.nonzero(~D[h, i])[0])


@pytest.mark.parametrize("fixture", ["tiny", "v8"])
def test_attention(fixture, request):
    layer = request.getfixturevalue(fixture)
    rng = np.random.default_rng(0)
    rows = [(h, i) for h in range(layer.H) for i in range(layer.nb)]
    if len(rows) > 400:
        idx = rng.choice(len(rows), 400, replace=False)
        rows = [rows[k] for k in sorted(idx)] + [(0, layer.nb - 1), (layer.H - 1, layer.nb - 2)]
    r = G.compare_attention(layer, rows)
    print(fixture, r)
    assert r["max_abs"] <= G.ATT_MAX_ABS and r["mean_rel"] <= G.ATT_MEAN_REL, r


@pytest.mark.parametrize("fixture", ["tiny", "v8"])
def test_bf16_output_is_rounded_f32_output(fixture, request):
    layer = request.getfixturevalue(fixture)
    assert torch.equal(layer.O32.to(torch.bfloat16).view(torch.int16), layer.buf.O.view(torch.int16))


def test_forward_equals_staged_calls(tiny):
    """The forward gives the staged calls' kept lists, best objectives and float32 output (the
    same ress_sparse_attn_f32 on the same CSR) bit for bit.  Its bf16 attention walks paired
    query blocks, whose one-sided blocks lead the lists, so a row takes its kept blocks in
    another order than over adjacent pairs: that output is checked against the oracle on
    every row (error beyond its bf16 rounding within the attention tolerance)."""
    layer, _ = layer_for("tiny_v2")
    layer.run_forward()
    assert np.array_equal(layer.csr()[1], tiny.csr()[1])
    assert np.array_equal(layer.output(), tiny.output())
    assert np.array_equal(layer.buf.J_best.cpu().numpy(), tiny.buf.J_best.cpu().numpy())
    r = G.compare_attention_bf16(layer, [(h, i) for h in range(layer.H) for i in range(layer.nq)])
    assert r["max_abs"] <= G.ATT_MAX_ABS and r["mean_rel"] <= G.ATT_MEAN_REL, r


def greedy_pairs(keep):
    """Greedy matching by weight of the query blocks of one window (host restatement of
    the pairing's definition): keep [n, nb] bool kept candidate sets; of all pairs of unpaired
    blocks the one sharing most kept blocks (clamped at 2047) is taken next, ties to the
    nearer pair, then to the lower first block.  Pairs (a, b), a < b, by ascending a."""
    n = keep.shape[0]
    ov = np.minimum(keep.astype(np.int64) @ keep.T.astype(np.int64), 2047)
    order = sorted(((int(ov[a, b]), -(b - a), -a, a, b) for a in range(n) for b in range(a + 1, n)),
                   reverse=True)
    free = np.ones(n, bool)
    pairs = []
    for *_, a, b in order:
        if free[a] and free[b]:
            free[a] = free[b] = False
            pairs.append((a, b))
    return sorted(pairs)


def item_list(la, lb):
    """The attention item list of two query blocks' kept lists (host restatement of the
    layout): the k-th block kept by the first only and the k-th kept by the second only
    (k below the smaller count, both ascending) at positions 2k, 2k + 1, then the rest of the
    union ascending; entry j | mask << 16 (bit 0: the first block keeps j, bit 1: the second)."""
    sa, sb = set(int(j) for j in la), set(int(j) for j in lb)
    only_a, only_b = sorted(sa - sb), sorted(sb - sa)
    P = min(len(only_a), len(only_b))
    out = []
    for k in range(P):
        out += [only_a[k] | (1 << 16), only_b[k] | (2 << 16)]
    lead = set(only_a[:P]) | set(only_b[:P])
    out += [j | ((int(j in sa) | (int(j in sb) << 1)) << 16) for j in sorted((sa | sb) - lead)]
    return np.asarray(out, dtype=np.int64)


@pytest.mark.parametrize("name,q_block", [("tiny_v2", 64), ("tiny_v2", 128), ("vggt_v8", 64),
                                          ("vggt_v8", 128), ("vggt_v32", 64)])
def test_forward_item_lists(name, q_block):
    """ress_forward's CSR kernel also writes the attention items' lists (entry j | mask << 16
    at each item's slot, the CSR offset of rows 2u, 2u + 1; lengths in plen).  On the 64-token
    grid the forward pairs the candidate query blocks within windows of 64 by the overlap of
    their kept lists (table prow): the items partition the rows, and each list is exactly the
    union of its two rows' lists with the right masks, laid out as the k-th block kept by the
    first row only and the k-th kept by the second only (k < P, the smaller count) at
    positions 2k, 2k + 1, then the rest in ascending order.  Rows take their blocks in list
    order, so the output over these pairs and the one over adjacent pairs (ress_sparse_attn
    on the same CSR) differ by rounding: both are within the attention tolerance of the
    exact result, and they are equal bit for bit on the 128-token grid, where both walk the
    same lists.  The pairing keeps fewer one-sided union entries than adjacent pairs,
    and is the greedy matching by overlap of the kept sets."""
    wl = synth.WORKLOADS[name]
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), wl.rounds, wl.rho,
                    q_block=q_block)
    r, b = layer.ress, layer.buf
    r.prepare_wo(layer.d, layer.W, b.F)
    r.forward(layer.d, layer.Q, layer.K, layer.V, b.F, layer.c_h, layer.rounds, layer.rho, b.ws,
              b.row_ptr, b.col_idx, b.O, b.J_best)
    r.status(b.ws)
    rpi = 1 if q_block == 128 else 2
    items = -(-layer.nq // rpi)
    npaired = layer.nqc // 2 if q_block == 64 else 0
    plen = layer.ws("plen", torch.int32)[:layer.H * items].copy()
    plist = layer.ws("t", torch.int32).copy()
    prow = layer.ws("prow", torch.int32)[:layer.H * items].copy()
    O_f = b.O.clone()
    rp, ci = layer.csr()
    kept = lambda h, i: ci[rp[h * layer.nq + i]:rp[h * layer.nq + i + 1]]
    entries = union = 0
    adjacent_union = 0
    for h in range(layer.H):
        seen = []
        for u in range(items):
            if u < npaired:
                ra, rb = int(prow[h * items + u]) & 0xffff, int(prow[h * items + u]) >> 16
                assert ra < rb and ra // 64 == rb // 64 == u // 32, (h, u, ra, rb)
                rows = [ra, rb]
            else:
                rows = [u] if rpi == 1 else [x for x in (2 * u, 2 * u + 1) if x < layer.nq]
            seen += rows
            la = kept(h, rows[0])
            lb = kept(h, rows[1]) if len(rows) > 1 else (la if rpi == 1 else np.zeros(0, int))
            want = item_list(la, lb)
            s0, n = rp[h * layer.nq + u * rpi], plen[h * items + u]
            got = plist[s0:s0 + n]
            assert n == len(want), (h, u)
            assert np.array_equal(got, want), (h, u)
            entries += len(la) + len(lb)
            union += n
            if u < npaired:  # the adjacent pair of the same slot, for comparison
                aa, ab = kept(h, 2 * u), kept(h, 2 * u + 1)
                adjacent_union += len(set(aa) | set(ab))
            elif rows:
                adjacent_union += n
        assert sorted(seen) == list(range(layer.nq)), h
    if npaired:
        print(name, "union efficiency", entries / 2 / union, "adjacent", entries / 2 / adjacent_union)
        assert union <= adjacent_union
        # the table is exactly the greedy matching by overlap of the best kept sets, window
        # by window, its pairs in the order of their first blocks
        drop = layer.drop_sets("bmask")
        cand = np.arange(layer.nb) < layer.ncand
        for h in range(layer.H):
            keep = ~drop[h] & cand
            for w0 in range(0, 2 * npaired, 64):
                n = min(64, 2 * npaired - w0)
                want = [(w0 + a, w0 + b) for a, b in greedy_pairs(keep[w0:w0 + n])]
                got = [(int(v) & 0xffff, int(v) >> 16)
                       for v in prow[h * items + w0 // 2:h * items + w0 // 2 + n // 2]]
                assert got == want, (h, w0)
    r.sparse_attn(layer.d, layer.Q, layer.K, layer.V, b.row_ptr, b.col_idx, b.O, b.ws)
    r.status(b.ws)
    if q_block == 128:
        assert torch.equal(O_f.view(torch.int16), b.O.view(torch.int16))
    else:
        # each within the tolerance of the exact result, beyond its rounding to bf16
        a, s = O_f.float(), b.O.float()
        assert bool(((a - s).abs() <= 2 * G.ATT_MAX_ABS + 2.0 ** -8 * (a.abs() + s.abs())).all())
        assert float((a - s).abs().mean() / s.abs().mean()) <= 2 * G.ATT_MEAN_REL
        b.O.copy_(O_f)
        rng = np.random.default_rng(7)
        rows = [(h, i) for h in range(layer.H) for i in range(layer.nq)]
        rows = [rows[k] for k in sorted(rng.choice(len(rows), min(len(rows), 200), replace=False))]
        r2 = G.compare_attention_bf16(layer, rows)
        assert r2["max_abs"] <= G.ATT_MAX_ABS and r2["mean_rel"] <= G.ATT_MEAN_REL, r2


def test_deterministic_bits():
    a, _ = layer_for("tiny_v2")
    b, _ = layer_for("tiny_v2")
    a.run()
    b.run()
    assert np.array_equal(a.csr()[1], b.csr()[1])
    assert torch.equal(a.buf.O.view(torch.int16), b.buf.O.view(torch.int16))
    assert torch.equal(a.buf.J_best, b.buf.J_best)


@pytest.mark.parametrize("N,H,ns,c,R", [
    (65, 1, 0, 1, 2),          # two blocks, one candidate, ragged tail
    (64 * 7, 1, 0, 3, 3),      # no special tokens, no ragged tail, odd block count
    (64 * 10 + 17, 3, 5, 4, 2),  # three heads, ragged tail with special tokens
    (1000, 2, 40, 1, 1),       # budget of one block
    (1300, 2, 7, 20, 3),       # c_h = |P|: nothing dropped (0% sparsity)
])
def test_edge_shapes(N, H, ns, c, R):
    inp = synth.make_random_layer(N, H, 64 * H, seed=N + H)
    nc = O.n_candidates(N, ns)
    c = min(c, nc)
    layer = G.Layer(inp, ns, [c] * H, R).run()
    sel = layer.oracle_select()
    r = G.compare_selection(layer, sel)
    G.check_selection(r)
    assert r["mismatched"] == 0, r
    rows = [(h, i) for h in range(H) for i in range(layer.nb)]
    a = G.compare_attention(layer, rows)
    assert a["max_abs"] <= G.ATT_MAX_ABS and a["mean_rel"] <= G.ATT_MEAN_REL, a


def test_dense_csr_is_dense_attention(tiny):
    """A CSR that keeps every block gives dense attention (same kernel, no dropped tiles)."""
    H, nb = tiny.H, tiny.nb
    rp = torch.arange(0, H * nb * nb + 1, nb, dtype=torch.int32, device="cuda")
    ci = torch.arange(nb, dtype=torch.int32, device="cuda").repeat(H * nb)
    O_ = torch.empty_like(tiny.O32)
    tiny.ress.sparse_attn_f32(tiny.d, tiny.Q, tiny.K, tiny.V, rp, ci, O_, tiny.buf.ws)
    tiny.ress.status(tiny.buf.ws)
    q, k, v = (t.float().permute(1, 0, 2) for t in (tiny.Q, tiny.K, tiny.V))
    ref = torch.nn.functional.scaled_dot_product_attention(q, k, v).permute(1, 0, 2)
    diff = (O_.float() - ref).abs()
    assert diff.max().item() <= G.ATT_MAX_ABS
    assert diff.sum().item() / ref.abs().sum().item() <= G.ATT_MEAN_REL


def _caller_csr(layer, kept):
    H, nq = layer.H, layer.nq
    lens = [len(kept[(h, i)]) for h in range(H) for i in range(nq)]
    rp = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32, device="cuda")
    ci = torch.tensor(np.concatenate([kept[(h, i)] for h in range(H) for i in range(nq)]),
                      dtype=torch.int32, device="cuda")
    return rp, ci


def _attn_f32(layer, kept):
    rp, ci = _caller_csr(layer, kept)
    out = torch.empty_like(layer.O32)
    layer.ress.sparse_attn_f32(layer.d, layer.Q, layer.K, layer.V, rp, ci, out, layer.buf.ws)
    layer.ress.status(layer.buf.ws)
    return out


def _bf16_p_bound(layer, kept, h, i):
    """Exact attention of query block (h, i) over its kept blocks (float64) and a bound on
    the kernel's error there: each probability is rounded to bf16 (8 significant bits,
    relative error at most u = 2^-8) and the row sum is formed from the same rounded values,
    so the output moves by at most u / (1 - u) sum_k w_k |v_k - o| <= 1.01 u (sum_k w_k |v_k|
    + |o|); 2^-12 sum_k w_k |v_k| more covers the float32 scores, exponentials and
    accumulations (about 2^-13 of it for 2,000 keys)."""
    Q, K, V = (G.widen(layer.bits[n]) for n in ("Q", "K", "V"))
    N = layer.N
    q = Q[i * 64:min(N, (i + 1) * 64), h].astype(np.float64)
    idx = np.concatenate([np.arange(j * 64, min(N, (j + 1) * 64)) for j in kept[(h, i)]])
    k, v = K[idx, h].astype(np.float64), V[idx, h].astype(np.float64)
    s = q @ k.T / 8.0
    w = np.exp(s - s.max(1, keepdims=True))
    w /= w.sum(1, keepdims=True)
    o = w @ v
    wv = w @ np.abs(v)
    return o, 1.01 * 2.0 ** -8 * (wv + np.abs(o)) + 2.0 ** -12 * wv


@pytest.mark.parametrize("case", ["disjoint", "leftover", "unequal"])
def test_one_sided_lists(tiny, case):
    """Caller lists in which the two query blocks of each adjacent pair keep (mostly) disjoint
    key blocks, so that most union entries are one-sided (the other block's rows get P = 0)
    and lead the list, alternating between the two blocks.  "disjoint": every entry is
    one-sided.  "leftover": three alternating pairs, then one-sided entries of the second
    block, shared blocks and the ragged last block.  In both every row still takes its blocks
    in ascending order, and its float32 output is bit for bit that of the same row given a
    partner with its own list (no one-sided entry at all): a row's result depends only on its
    own blocks and their order.  "unequal": a third of the blocks against the rest, where the
    alternation reorders rows' blocks.  In all three the output is within the bound of bf16
    probability rounding of the exact attention, the bf16 output is the rounding of the
    float32 one, and the lists k_pairs builds follow item_list's layout."""
    H, nb, nq = tiny.H, tiny.nb, tiny.nq
    kept = {}
    for h in range(H):
        for i in range(nq):
            if case == "disjoint":
                ks = [j for j in range(nb - 1) if j % 2 == (i + h) % 2]
            elif case == "leftover":
                ks = ([1, 3, 5, nb - 3, nb - 2] if i % 2 == 0
                      else list(range(0, nb - 4, 2)) + [nb - 3, nb - 2, nb - 1])
            elif i % 2 == 0:
                ks = [j for j in range(nb - 1) if j % 3 == 0]
            else:
                ks = [0] + [j for j in range(nb) if j % 3 != 0]
            kept[(h, i)] = np.asarray(sorted(ks), dtype=np.int64)
    got = _attn_f32(tiny, kept)
    # the union lists k_pairs wrote for the adjacent pairs (2p, 2p + 1) of each head
    plist = tiny.ws("t", torch.int32)
    npairs = (nq + 1) // 2
    plen = tiny.ws("plen", torch.int32)[:H * npairs]
    offs = np.concatenate([[0], np.cumsum([len(kept[(h, i)]) for h in range(H) for i in range(nq)])])
    for h in range(H):
        for pp in range(npairs):
            lb = kept[(h, 2 * pp + 1)] if 2 * pp + 1 < nq else np.zeros(0, np.int64)
            want = item_list(kept[(h, 2 * pp)], lb)
            s0 = offs[h * nq + 2 * pp]
            assert plen[h * npairs + pp] == len(want), (h, pp)
            assert np.array_equal(plist[s0:s0 + len(want)], want), (h, pp)
    rp, ci = _caller_csr(tiny, kept)
    O16 = torch.empty_like(tiny.buf.O)
    tiny.ress.sparse_attn(tiny.d, tiny.Q, tiny.K, tiny.V, rp, ci, O16, tiny.buf.ws)
    tiny.ress.status(tiny.buf.ws)
    assert torch.equal(got.to(torch.bfloat16).view(torch.int16), O16.view(torch.int16))
    got = got.cpu().numpy()
    if case != "unequal":
        alone = np.empty_like(got)
        for par in (0, 1):  # rows of parity par, each sharing its tile with a copy of its list
            same = {(h, i): kept[(h, min(nq - 1, i - i % 2 + par))] for h in range(H) for i in range(nq)}
            o = _attn_f32(tiny, same).cpu().numpy()
            for i in range(par, nq, 2):
                alone[i * 64:(i + 1) * 64] = o[i * 64:(i + 1) * 64]
        assert np.array_equal(got.view(np.uint32), alone.view(np.uint32))
    for h in range(H):
        for i in range(nq):
            o, bound = _bf16_p_bound(tiny, kept, h, i)
            g = got[i * 64:i * 64 + o.shape[0], h, :]
            assert np.all(np.abs(g - o) <= bound), (h, i, float(np.abs(g - o).max()))


def test_bad_csr_index_is_reported_not_faulted(tiny):
    import paper_2609_35593_gb300 as ress
    rp = tiny.buf.row_ptr.clone()
    ci = tiny.buf.col_idx.clone()
    ci[5] = tiny.nb + 100
    O_ = torch.empty_like(tiny.buf.O)
    ress.sparse_attn(tiny.d, tiny.Q, tiny.K, tiny.V, rp, ci, O_, tiny.buf.ws)
    with pytest.raises(ress.RessError) as e:
        ress.status(tiny.buf.ws)
    assert e.value.code == -6
    ress.status(tiny.buf.ws)  # cleared


def test_headline_shape_sampled():
    """32 views, 16 heads, 90% sparsity, R = 3: sampled rows against the oracle, and
    properties that hold at any size on every row."""
    layer, wl = layer_for("vggt_v32")
    layer.run()
    rng = np.random.default_rng(1)
    rows = [(int(h), int(i)) for h, i in zip(rng.integers(0, wl.heads, 24), rng.integers(0, wl.n_candidates, 24))]
    sel = layer.oracle_select(rows)
    r = G.compare_selection(layer, sel)
    G.check_selection(r)
    print(r)
    assert r["mismatched"] == 0, r
    J0 = layer.ws("J0", shape=(layer.H, layer.nb))
    Jb = layer.buf.J_best.cpu().numpy().reshape(layer.H, layer.nb)
    assert np.all(Jb[:, :layer.ncand] <= J0[:, :layer.ncand])
    rp, ci = layer.csr()
    assert rp[-1] == ci.size
    arows = rows[:8] + [(0, layer.nb - 1), (5, layer.nb - 2)]
    a = G.compare_attention(layer, arows)
    print(a)
    assert a["max_abs"] <= G.ATT_MAX_ABS and a["mean_rel"] <= G.ATT_MEAN_REL, a


def test_attention_rescale_path():
    """Logits that grow along every kept list by several times the lazy-rescale threshold
    (2^20 in the exp2 domain), so the kernel rescales its accumulator several times per row;
    the output must still match the oracle."""
    N, H, ns, c, R = 64 * 24 + 5, 2, 5, 12, 2
    inp = synth.make_random_layer(N, H, 64 * H, seed=11)
    rng = np.random.default_rng(5)
    q = synth.bf16_to_f32(inp["Q"])
    k = synth.bf16_to_f32(inp["K"])
    u = rng.standard_normal((H, 64)).astype(np.float32)
    blk = np.minimum(np.arange(N) // 64, (N - ns) // 64).astype(np.float32)
    q = q + 2.0 * u[None]                                  # every query leans along u
    k = k + (0.3 * blk)[:, None, None] * u[None]           # keys along u grow with the block
    inp = dict(inp, Q=synth.bf16_bits(q), K=synth.bf16_bits(k))
    layer = G.Layer(inp, ns, [c] * H, R).run()
    # the exp2-domain growth of the running block max along each kept list, from the
    # inputs the kernel received: at least one rescale per sampled row must be needed
    kq, kk = synth.bf16_to_f32(inp["Q"]), synth.bf16_to_f32(inp["K"])
    kept = layer.kept()
    scale = 1.4426950408889634 / 8.0
    rescales = 0
    rows = [(h, i) for h in range(H) for i in range(layer.nb)]
    for (h, i) in rows:
        qi = kq[64 * i:64 * i + 64, h]
        m_use = None
        for j in kept[(h, i)]:
            mt = float((qi @ kk[64 * j:64 * j + 64, h].T).max(axis=1).min()) * scale
            if m_use is None:
                m_use = mt
            elif mt > m_use + 20.0:
                m_use, rescales = mt, rescales + 1
    assert rescales > len(rows)  # several rescales per row on average
    a = G.compare_attention(layer, rows)
    assert a["max_abs"] <= G.ATT_MAX_ABS and a["mean_rel"] <= G.ATT_MEAN_REL, a


@pytest.mark.parametrize("name,kw", [
    ("vggt_v100", {}),                                  # 137400 tokens, cross-view term
    ("vggt_v64", {"sparsity": 0.5, "rounds": 4}),       # sweep corners
    ("vggt_v64", {"sparsity": 0.95, "rounds": 0}),
])
def test_large_shapes_sampled(name, kw):
    """The long-view configuration and two corners of the 64-view sweep: sampled rows
    against the oracle, and the properties that hold at any size on every row."""
    layer, wl = layer_for(name, **kw)
    layer.run()
    rng = np.random.default_rng(2)
    rows = [(int(h), int(i)) for h, i in zip(rng.integers(0, wl.heads, 10), rng.integers(0, wl.n_candidates, 10))]
    r = G.compare_selection(layer, layer.oracle_select(rows))
    G.check_selection(r)
    print(name, kw, r)
    assert r["mismatched"] == 0, r
    J0 = layer.ws("J0", shape=(layer.H, layer.nb))
    Jb = layer.buf.J_best.cpu().numpy().reshape(layer.H, layer.nb)
    assert np.all(Jb[:, :layer.ncand] <= J0[:, :layer.ncand])
    if wl.rounds == 0:
        assert np.array_equal(Jb[:, :layer.ncand], J0[:, :layer.ncand])
    rp, ci = layer.csr()
    assert rp[-1] == ci.size
    arows = rows[:6] + [(0, layer.nb - 1), (wl.heads - 1, layer.nb - 2)]
    a = G.compare_attention(layer, arows)
    print(a)
    assert a["max_abs"] <= G.ATT_MAX_ABS and a["mean_rel"] <= G.ATT_MEAN_REL, a


def test_maximum_shape_sampled():
    """The largest sequence the library takes (RESS_MAX_BLOCKS = 4096 key blocks, 262,144
    tokens; 2 heads): a budget above 128 per row (the all-keys selection of the score
    kernel) and a first round with m > 64 (the bitmask path of the rounds).  Sampled rows of
    the selection and of the attention against the oracle, and the invariants on every row."""
    N, H, ns = 64 * 4096, 2, 5
    inp = synth.make_random_layer(N, H, 64 * H, seed=4096)
    nc = O.n_candidates(N, ns)
    c = int(round(0.1 * nc))
    layer = G.Layer(inp, ns, [c] * H, 2).run()
    assert layer.nb == 4096 and layer.ncand == nc
    rng = np.random.default_rng(3)
    rows = [(int(h), int(i)) for h, i in zip(rng.integers(0, H, 6), rng.integers(0, nc, 6))]
    r = G.compare_selection(layer, layer.oracle_select(rows + [(H - 1, nc - 1)]))
    G.check_selection(r)
    assert r["mismatched"] == 0, r
    assert r["worst_row_rel"] <= G.DRIFT_REL, r
    J0 = layer.ws("J0", shape=(H, layer.nb))
    Jb = layer.buf.J_best.cpu().numpy().reshape(H, layer.nb)
    assert np.all(Jb[:, :nc] <= J0[:, :nc])
    rp, ci = layer.csr()
    assert rp[-1] == ci.size == H * (nc * (c + layer.nb - nc) + (layer.nb - nc) * layer.nb)
    a = G.compare_attention(layer, rows[:4] + [(0, layer.nb - 1)])
    assert a["max_abs"] <= G.ATT_MAX_ABS and a["mean_rel"] <= G.ATT_MEAN_REL, a


@pytest.mark.parametrize("q_block", [64, 128])
def test_equal_keys_keep_the_lowest_indices(q_block):
    """Ties: with every key token equal, every pooled probability of a row is the same, so
    the probability rule keeps the c_h candidates of lowest index (the tie order of Eq. 7's
    top-c in this build and in the oracle) on every row; the rounds then follow the oracle."""
    N, H, ns = 64 * 40, 2, 5
    inp = synth.make_random_layer(N, H, 64 * H, seed=40)
    inp["K"][:] = inp["K"][0:1]
    nc = O.n_candidates(N, ns)
    c = 11
    layer = G.Layer(inp, ns, [c] * H, 0, variant=O.Variant(key="probability"),
                    q_block=q_block).run(attention=False)
    D = layer.drop_sets()
    want = np.ones(layer.nb, dtype=bool)
    want[:c] = False
    want[nc:] = False
    for h in range(H):
        for i in range(layer.nqc):
            assert np.array_equal(D[h, i], want), (h, i)
    layer3 = G.Layer(inp, ns, [c] * H, 3, variant=O.Variant(key="probability"),
                     q_block=q_block).run(attention=False)
    r = G.compare_selection(layer3, layer3.oracle_select())
    G.check_selection(r)
    assert r["mismatched"] == 0, r


@pytest.mark.parametrize("name,q_block", [("tiny_v2", 64), ("tiny_v2", 128), ("vggt_v8", 64)])
def test_forward_host_equals_forward(name, q_block):
    """ress_forward_host (copies in, selection, then the attention in chunks of query rows
    whose output rows are copied out as each chunk completes, on library streams joined back
    into the caller's) gives the bits of the device forward, and the caller's stream alone
    orders the result: every output row is on the host once that stream is done."""
    wl = synth.WORKLOADS[name]
    ref = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), wl.rounds, wl.rho,
                  q_block=q_block).run_forward()
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), wl.rounds, wl.rho,
                    q_block=q_block)
    r, b = layer.ress, layer.buf
    r.prepare_wo(layer.d, layer.W, b.F)
    torch.cuda.synchronize()
    Qh, Kh, Vh = (t.cpu().pin_memory() for t in (layer.Q, layer.K, layer.V))
    Oh = torch.empty(b.O.shape, dtype=torch.bfloat16).pin_memory()
    Oh.view(torch.int16).fill_(-1)  # NaN bits: a row the copies miss stays visible
    Qd, Kd, Vd, Od = (torch.empty_like(t) for t in (layer.Q, layer.K, layer.V, b.O))
    s = torch.cuda.Stream()
    for _ in range(2):  # the second call reuses the library's streams and events
        r.forward_host(layer.d, Qh, Kh, Vh, Oh, Qd, Kd, Vd, Od, b.F, layer.c_h, layer.rounds,
                       layer.rho, b.ws, b.row_ptr, b.col_idx, b.J_best, stream=s)
        s.synchronize()
        assert torch.equal(Oh.view(torch.int16), ref.buf.O.cpu().view(torch.int16))
        Oh.view(torch.int16).fill_(-1)
    r.status(b.ws, stream=s)
    assert np.array_equal(layer.csr()[1], ref.csr()[1])


@pytest.mark.parametrize("fixture_name", ["tiny_v2", "vggt_v8"])
def test_gain_products(fixture_name):
    """Restoration gains t_ij = (y~_i - z~_j) . g~_i (Eq. 14/15), computed on the tensor
    cores from three-term bf16 splits, against float64 products of the same float32 y~, z~
    and g~ (the state after the initial selection, i.e. the start of round 0)."""
    layer, wl = layer_for(fixture_name)
    r, b = layer.ress, layer.buf
    r.prepare_wo(layer.d, layer.W, b.F)
    r.score(layer.d, layer.Q, layer.K, layer.V, b.F, layer.c_h, b.ws)
    torch.cuda.synchronize()
    H, nb, nc, L = layer.H, layer.nb, layer.ncand, b.layout
    y = layer.ws("ytil", shape=(H, nb, 64)).astype(np.float64)
    z = layer.ws("ztil", shape=(H, nb, 64)).astype(np.float64)
    g = layer.ws("gtil", shape=(H, nb, 64)).astype(np.float64)
    cdot = layer.ws("cdot", shape=(H, nb)).astype(np.float64)
    for name, x, rows in (("asplit", g, nc), ("zsplit", z, nb)):
        terms = synth.bf16_to_f32(layer.ws(name, torch.int16, (3, H, nb, 64)).view(np.uint16))
        hi, mid, lo = (terms[k].astype(np.float64)[:, :rows] for k in range(3))
        xs = x[:, :rows]
        assert np.all(np.abs(mid) <= 2.0 ** -8 * np.abs(xs) + 1e-30)
        assert np.all(np.abs(hi + mid + lo - xs) <= 2.0 ** -23 * np.abs(xs) + 1e-30), name
    yn, zn, gn = (np.linalg.norm(v, axis=2) for v in (y, z, g))
    np.testing.assert_array_less(np.abs(cdot[:, :nc] - (y * g).sum(2)[:, :nc]),
                                 1e-5 * (yn * gn)[:, :nc] + 1e-30)
    r.restore(layer.d, layer.c_h, 1, layer.rho, b.ws, b.row_ptr, b.col_idx, b.J_best)
    r.status(b.ws)
    torch.cuda.synchronize()
    t = layer.ws("t", shape=(H, nb, L.ld))
    checked = 0
    for h in range(H):
        if min(O.swap_schedule(layer.c_h[h], 1, layer.rho)[0], nc - layer.c_h[h]) <= 0:
            continue
        ref = (y[h, :nc] * g[h, :nc]).sum(1)[:, None] - g[h, :nc] @ z[h, :nc].T
        bound = 1e-5 * gn[h, :nc, None] * (yn[h, :nc, None] + zn[h, None, :nc]) + 1e-30
        err = np.abs(t[h, :nc, :nc] - ref)
        assert np.all(err <= bound), (h, float((err / bound).max()))
        checked += 1
    assert checked > 0


@pytest.mark.parametrize("fixture_name", ["tiny_v2", "vggt_v8"])
def test_tensor_core_scoring(fixture_name):
    """Pooled map P, y~ and q (Sec. 4.1, Eq. 1, Eq. 9), computed on the tensor cores from
    three-term bf16 splits, against float64 arithmetic on the same float32 pooled vectors
    q_bar, k_bar and z~ that the GPU produced."""
    layer, wl = layer_for(fixture_name)
    r, b = layer.ress, layer.buf
    r.prepare_wo(layer.d, layer.W, b.F)
    r.score(layer.d, layer.Q, layer.K, layer.V, b.F, layer.c_h, b.ws)
    r.status(b.ws)
    torch.cuda.synchronize()
    H, nb, nc, L = layer.H, layer.nb, layer.ncand, b.layout
    qb = layer.ws("qbar", shape=(H, nb, 64)).astype(np.float64)
    kb = layer.ws("kbar", shape=(H, nb, 64)).astype(np.float64)
    z = layer.ws("ztil", shape=(H, nb, 64)).astype(np.float64)
    y = layer.ws("ytil", shape=(H, nb, 64)).astype(np.float64)
    P = layer.ws("P", shape=(H, nb, L.ld))
    q = layer.ws("q", shape=(H, nb, L.ld))
    nz = layer.ws("nz", shape=(H, nb)).astype(np.float64)
    np.testing.assert_allclose(nz, (z * z).sum(2), rtol=1e-5)
    for h in range(H):
        logit = qb[h, :nc] @ kb[h].T / 8.0
        Pr = np.exp(logit - logit.max(1, keepdims=True))
        Pr /= Pr.sum(1, keepdims=True)
        np.testing.assert_allclose(P[h, :nc, :nb], Pr, rtol=2e-5, atol=1e-7 * Pr.max())
        assert np.all(P[h, :nc, nb:L.ld] == 0)
        yr = Pr @ z[h]
        yn = np.linalg.norm(yr, axis=1, keepdims=True)
        assert np.all(np.abs(y[h, :nc] - yr) <= 1e-5 * (yn + np.abs(yr)) + 1e-30)
        # q from the GPU's own y~ (its rounding is not q's error)
        qr = ((y[h, :nc, None, :] - z[h, None, :, :]) ** 2).sum(2)
        scale = (y[h, :nc] ** 2).sum(1)[:, None] + nz[h][None, :]
        assert np.all(np.abs(q[h, :nc, :nb] - qr) <= 2e-6 * scale + 1e-30), h
        assert np.all(q[h, :nc, :nb] >= 0)


def test_kernel_launch_counter():
    """ress_kernel_launches counts every kernel of a forward: six for scoring (pooling,
    z-projection, logits, P with y~, q, score rows), two per restoration round, the pairing
    of the query blocks, the CSR kernel (which also writes the attention items' lists) and
    the attention kernel."""
    layer, wl = layer_for("tiny_v2")
    r, b = layer.ress, layer.buf
    r.prepare_wo(layer.d, layer.W, b.F)
    n0 = r.kernel_launches()
    r.forward(layer.d, layer.Q, layer.K, layer.V, b.F, layer.c_h, layer.rounds, layer.rho, b.ws,
              b.row_ptr, b.col_idx, b.O, b.J_best)
    torch.cuda.synchronize()
    assert r.kernel_launches() - n0 == 6 + 2 * layer.rounds + 1 + 1 + 1


def test_large_swap_count_parity():
    """A budget of 135 of |P| = 171 candidates on the 8-view layer: a first swap count of 33,
    more survivors than lanes in the round kernel's selection (its radix path), every row
    against the oracle."""
    wl = synth.WORKLOADS["vggt_v8"]
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, [135] * wl.heads, wl.rounds,
                    wl.rho).run(attention=False)
    assert O.swap_schedule(135, 1, wl.rho)[0] == 33
    r = G.compare_selection(layer, layer.oracle_select())
    G.check_selection(r)
    assert r["exact"] >= 0.95 * (r["exact"] + r["near"]), r


def _bf16_tensor(a):
    """float array -> (device bf16 tensor, the float64 values it holds)."""
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16)
    return t.cuda(), t.float().numpy().astype(np.float64)


@pytest.mark.parametrize("fixture", ["tiny", "v8"])
def test_out_proj_residual_update(fixture, request):
    """y = x + O W_o^T (Sec. 3) on the tensor cores against float64 on the same bf16 inputs:
    the attention output of the layer, a random residual x; also x = NULL and in place."""
    layer = request.getfixturevalue(fixture)
    N, Dm = layer.N, layer.d_model
    rng = np.random.default_rng(11)
    x, xf = _bf16_tensor(rng.normal(size=(N, Dm)))
    Of = layer.buf.O.float().cpu().numpy().reshape(N, -1).astype(np.float64)
    Wf = layer.W_o()
    ref = O.residual_update(xf, Of, Wf)
    scale = np.abs(Of) @ np.abs(Wf).T + np.abs(xf)  # bound of the accumulated magnitudes
    y = torch.empty(N, Dm, dtype=torch.bfloat16, device="cuda")
    layer.ress.out_proj(layer.d, layer.buf.O, layer.W, x, y, layer.buf.ws)
    layer.ress.status(layer.buf.ws)
    got = y.float().cpu().numpy()
    assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 1e-5 * scale + 1e-6)
    y0 = torch.empty_like(y)
    layer.ress.out_proj(layer.d, layer.buf.O, layer.W, None, y0, layer.buf.ws)
    ref0 = O.residual_update(None, Of, Wf)
    assert np.all(np.abs(y0.float().cpu().numpy() - ref0) <= 2.0 ** -8 * np.abs(ref0) + 1e-5 * scale + 1e-6)
    xi = x.clone()
    layer.ress.out_proj(layer.d, layer.buf.O, layer.W, xi, xi, layer.buf.ws)  # in place
    torch.cuda.synchronize()
    assert torch.equal(xi.view(torch.int16), y.view(torch.int16))


@pytest.mark.parametrize("fixture", ["tiny", "v8"])
def test_token_drift_sparse_vs_dense(fixture, request):
    """Sec. 3's token-level drift per query block, ||W_o (O_sparse - O_dense)||^2 over the
    block's tokens, on the tensor cores against float64 on the same bf16 outputs."""
    layer = request.getfixturevalue(fixture)
    H, nb, N = layer.H, layer.nb, layer.N
    rp = torch.arange(0, H * nb * nb + 1, nb, dtype=torch.int32, device="cuda")
    ci = torch.arange(nb, dtype=torch.int32, device="cuda").repeat(H * nb)
    O_dense = torch.empty_like(layer.buf.O)
    layer.ress.sparse_attn(layer.d, layer.Q, layer.K, layer.V, rp, ci, O_dense, layer.buf.ws)
    drift = torch.empty(nb, dtype=torch.float32, device="cuda")
    layer.ress.token_drift(layer.d, layer.buf.O, O_dense, layer.W, drift, layer.buf.ws)
    layer.ress.status(layer.buf.ws)
    got = drift.cpu().numpy().astype(np.float64)
    Oa = layer.buf.O.float().cpu().numpy().reshape(N, -1)
    Ob = O_dense.float().cpu().numpy().reshape(N, -1)
    ref = O.token_drift(Oa, Ob, layer.W_o())
    ya, yb = (O.residual_update(None, o, layer.W_o()) for o in (Oa, Ob))
    mag = np.array([float((ya[64 * b: 64 * (b + 1)] ** 2).sum() + (yb[64 * b: 64 * (b + 1)] ** 2).sum())
                    for b in range(nb)])
    assert np.all(np.abs(got - ref) <= 1e-4 * ref + 1e-6 * mag + 1e-12), np.max(np.abs(got - ref) / (ref + 1e-30))
    assert np.all(got[layer.ncand:] <= 1e-6 * mag[layer.ncand:] + 1e-12)  # special rows are dense


@pytest.mark.parametrize("name", ["tiny_v2", "vggt_v8"])
@pytest.mark.parametrize("variant,rounds", [
    (O.Variant(key="probability"), 0),     # top-k by pooled mass (Table 3's probability rule)
    (O.Variant(key="probability"), 3),     # the same set refined by restoration
    (O.Variant(key="random", seed=5), 0),  # random selection (Fig. 8)
    (O.Variant(key="random", seed=5), 2),
    (O.Variant(maximize="swap"), 3),       # sign flip in the rounds only (Fig. 8, swap only)
    (O.Variant(maximize="full"), 3),       # sign flip from the initial selection (Fig. 8, full)
])
def test_selection_variants(name, variant, rounds):
    """The ablation variants of the selection against the oracle's: identical drop sets on
    every row outside the decision margin, drift within 1e-3."""
    wl = synth.WORKLOADS[name]
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), rounds, wl.rho,
                    variant=variant).run(attention=False)
    r = G.compare_selection(layer, layer.oracle_select())
    G.check_selection(r)
    assert r["mismatched"] == 0, r
    assert r["exact"] >= 0.95 * (r["exact"] + r["near"]), r
    assert r["worst_row_rel"] <= G.DRIFT_REL and r["sum_rel_gpu_vs_oracle"] <= G.DRIFT_REL, r


@pytest.mark.parametrize("name", ["tiny_v2", "vggt_v8"])
@pytest.mark.parametrize("variant,rounds", [
    (O.Variant(key="probability"), 3),
    (O.Variant(key="random", seed=11), 2),
    (O.Variant(maximize="swap"), 3),
    (O.Variant(maximize="full"), 3),
])
def test_selection_variants_paper_grid(name, variant, rounds):
    """The ablation variants on the paper's grid (128-token query blocks): identical drop
    sets outside the decision margin, drift within 1e-3."""
    wl = synth.WORKLOADS[name]
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), rounds, wl.rho,
                    variant=variant, q_block=128).run(attention=False)
    r = G.compare_selection(layer, layer.oracle_select())
    G.check_selection(r)
    assert r["mismatched"] == 0, r
    assert r["exact"] >= 0.95 * (r["exact"] + r["near"]), r
    assert r["worst_row_rel"] <= G.DRIFT_REL and r["sum_rel_gpu_vs_oracle"] <= G.DRIFT_REL, r


def test_cdf_threshold_headline_shape_sampled():
    """The CDF threshold at the 32-view headline shape: sampled rows of the drop sets against
    the oracle, and every CSR row exactly the complement of its drop set."""
    wl = synth.WORKLOADS["vggt_v32"]
    variant = O.Variant(key="probability", cdf=0.9)
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), 0, wl.rho,
                    variant=variant).run(attention=False)
    rng = np.random.default_rng(7)
    rows = [(int(h), int(i)) for h, i in zip(rng.integers(0, layer.H, 40),
                                             rng.integers(0, layer.nqc, 40))]
    r = G.compare_selection(layer, layer.oracle_select(rows))
    G.check_selection(r)
    assert r["mismatched"] == 0, r
    assert r["worst_row_rel"] <= G.DRIFT_REL, r
    rp, ci = layer.csr()
    D = layer.drop_sets()
    assert rp[-1] == int((~D[:, :layer.nqc]).sum()) + layer.H * (layer.nq - layer.nqc) * layer.nb
    for h, i in rows:
        k = ci[rp[h * layer.nq + i]:rp[h * layer.nq + i + 1]]
        assert np.array_equal(k, np.nonzero(~D[h, i])[0])


@pytest.mark.parametrize("name,q_block", [("tiny_v2", 64), ("vggt_v8", 64), ("vggt_v8", 128)])
@pytest.mark.parametrize("variant", [
    O.Variant(key="probability", cdf=0.9),  # SparseVGGT's rule: top-k plus the CDF threshold
    O.Variant(key="probability", cdf=0.5),
    O.Variant(cdf=0.8),                     # the drift key with the threshold on top
    O.Variant(key="random", seed=3, cdf=0.7),
])
def test_cdf_threshold_variant(name, q_block, variant):
    """CDF threshold (Table 3): drop sets against the oracle row by row, variable-length
    CSR rows (a device-side scan of the kept counts) that list exactly the kept blocks, the
    kept mass of every row at least tau unless the row keeps everything, and attention over
    those lists against the oracle on sampled rows."""
    wl = synth.WORKLOADS[name]
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), 0, wl.rho,
                    variant=variant, q_block=q_block).run()
    sel = layer.oracle_select()
    r = G.compare_selection(layer, sel)
    G.check_selection(r)
    assert r["mismatched"] == 0, r
    assert r["exact"] >= 0.95 * (r["exact"] + r["near"]), r
    assert r["worst_row_rel"] <= G.DRIFT_REL and r["sum_rel_gpu_vs_oracle"] <= G.DRIFT_REL, r
    rp, ci = layer.csr()
    D = layer.drop_sets()
    P = layer.ws("P", shape=(layer.H, layer.nq, layer.buf.layout.ld))
    lengths = np.diff(rp)
    assert rp[0] == 0 and np.all(lengths >= 1) and rp[-1] <= ci.size
    for h in range(layer.H):
        for i in range(layer.nq):
            k = ci[rp[h * layer.nq + i]:rp[h * layer.nq + i + 1]]
            if i >= layer.nqc:
                assert k.tolist() == list(range(layer.nb))
                continue
            assert np.array_equal(k, np.nonzero(~D[h, i])[0])
            assert k.size >= layer.c_h[h] + layer.nb - layer.ncand
            mass = float(P[h, i, k].astype(np.float64).sum())
            assert mass >= variant.cdf - 1e-4 or k.size == layer.nb, (h, i, mass)
    # the rule lengthens rows on the GPU exactly when it does in the oracle
    fixed = np.array([layer.c_h[h] + layer.nb - layer.ncand for h in range(layer.H)])
    gpu_ext = [lengths[h * layer.nq:h * layer.nq + layer.nqc].max() > fixed[h] for h in range(layer.H)]
    ora_ext = [any((~sel[(h, i)].D_best).sum() > fixed[h] for i in range(layer.nqc))
               for h in range(layer.H)]
    assert gpu_ext == ora_ext
    rows = [(h, i) for h in range(layer.H) for i in range(layer.nq)]
    if len(rows) > 60:
        idx = np.random.default_rng(2).choice(len(rows), 40, replace=False)
        rows = [rows[k] for k in sorted(idx)] + [(layer.H - 1, layer.nq - 1)]
    a = G.compare_attention(layer, rows)
    assert a["max_abs"] <= G.ATT_MAX_ABS and a["mean_rel"] <= G.ATT_MEAN_REL, a


def test_timed_out_wait_is_reported_and_context_stays_usable(tiny):
    """Failure detection without a fault: a kernel's bounded wait on a barrier that nothing
    completes gives up after its limit, the status word reports RESS_ETIMEOUT once (then is
    clear), and the next forward on the same context gives the same bits as before."""
    import paper_2609_35593_gb300 as ress
    layer, _ = layer_for("tiny_v2")
    r, b = layer.ress, layer.buf
    layer.run_forward()
    before = b.O.clone()
    r.wait_selftest(b.ws, 20000)
    with pytest.raises(ress.RessError) as e:
        r.status(b.ws)
    assert e.value.code == -5
    r.status(b.ws)  # cleared
    r.forward(layer.d, layer.Q, layer.K, layer.V, b.F, layer.c_h, layer.rounds, layer.rho, b.ws,
              b.row_ptr, b.col_idx, b.O, b.J_best)
    r.status(b.ws)
    assert torch.equal(b.O.view(torch.int16), before.view(torch.int16))


def test_invalid_variant_is_rejected(tiny):
    import paper_2609_35593_gb300 as ress
    bad = ress.Variant(7, 0, 0)
    with pytest.raises(ress.RessError) as e:
        ress.score(tiny.d, tiny.Q, tiny.K, tiny.V, tiny.buf.F, tiny.c_h, tiny.buf.ws, variant=bad)
    assert e.value.code == -1


@pytest.mark.parametrize("name", ["tiny_v2", "vggt_v8"])
def test_paper_grid_query_block_128(name):
    """The paper's own grid (Appendix F): 128-token query blocks over 64-token key blocks.
    Selection against the oracle on that grid, the CSR's row structure, and attention of
    every (sampled) query block against the oracle over the GPU's kept lists."""
    wl = synth.WORKLOADS[name]
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), wl.rounds, wl.rho,
                    q_block=128).run()
    assert layer.nq == -(-layer.N // 128)
    r = G.compare_selection(layer, layer.oracle_select())
    G.check_selection(r)
    assert r["mismatched"] == 0, r
    assert r["exact"] >= 0.95 * (r["exact"] + r["near"]), r
    assert r["worst_row_rel"] <= G.DRIFT_REL and r["sum_rel_gpu_vs_oracle"] <= G.DRIFT_REL, r
    rp, ci = layer.csr()
    D = layer.drop_sets()
    assert rp.size == layer.H * layer.nq + 1 and rp[-1] == ci.size
    for h in range(layer.H):
        for i in range(layer.nq):
            k = ci[rp[h * layer.nq + i]:rp[h * layer.nq + i + 1]]
            if i >= layer.nqc:
                assert k.tolist() == list(range(layer.nb))
            else:
                assert k.size == layer.c_h[h] + layer.nb - layer.ncand
                assert np.array_equal(k, np.nonzero(~D[h, i])[0])
    rows = [(h, i) for h in range(layer.H) for i in range(layer.nq)]
    if len(rows) > 60:
        idx = np.random.default_rng(1).choice(len(rows), 48, replace=False)
        rows = [rows[k] for k in sorted(idx)] + [(0, layer.nq - 1), (layer.H - 1, layer.nqc - 1)]
    a = G.compare_attention(layer, rows)
    assert a["max_abs"] <= G.ATT_MAX_ABS and a["mean_rel"] <= G.ATT_MEAN_REL, a


@pytest.mark.parametrize("N,H,ns,c,R", [
    (100, 1, 0, 1, 1),          # one ragged query block, two key blocks
    (64 * 9 + 30, 2, 40, 3, 2),  # special tokens straddling the last query blocks
    (1300, 2, 7, 20, 3),         # nothing dropped
])
def test_paper_grid_edge_shapes(N, H, ns, c, R):
    inp = synth.make_random_layer(N, H, 64 * H, seed=N + 7 * H)
    nc = O.n_candidates(N, ns)
    c = min(c, nc)
    layer = G.Layer(inp, ns, [c] * H, R, q_block=128).run()
    r = G.compare_selection(layer, layer.oracle_select())
    G.check_selection(r)
    assert r["mismatched"] == 0, r
    a = G.compare_attention(layer, [(h, i) for h in range(H) for i in range(layer.nq)])
    assert a["max_abs"] <= G.ATT_MAX_ABS and a["mean_rel"] <= G.ATT_MEAN_REL, a


def test_paper_grid_headline_shape_sampled():
    """The 32-view headline layer on the paper's grid (128-token query blocks): sampled rows
    of the selection and of the attention against the oracle, and J_best <= J0 on every
    sparsified row."""
    wl = synth.WORKLOADS["vggt_v32"]
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, wl.budgets(), wl.rounds, wl.rho,
                    q_block=128).run()
    rng = np.random.default_rng(2)
    rows = [(int(h), int(i)) for h, i in zip(rng.integers(0, wl.heads, 20), rng.integers(0, layer.nqc, 20))]
    r = G.compare_selection(layer, layer.oracle_select(rows))
    G.check_selection(r)
    assert r["mismatched"] == 0, r
    J0 = layer.ws("J0", shape=(layer.H, layer.nq))
    Jb = layer.buf.J_best.cpu().numpy().reshape(layer.H, layer.nq)
    assert np.all(Jb[:, :layer.nqc] <= J0[:, :layer.nqc])
    a = G.compare_attention(layer, rows[:8] + [(0, layer.nq - 1), (7, layer.nqc - 1)])
    assert a["max_abs"] <= G.ATT_MAX_ABS and a["mean_rel"] <= G.ATT_MEAN_REL, a


# ---------------------------------------------------------------------------------------
# Head-wise budgets (Sec. 4.4): a different c_h per head
# ---------------------------------------------------------------------------------------
UNEQUAL_BUDGETS = {
    # tiny_v2, |P| = 42: one block, every candidate (nothing dropped), the uniform budget, few
    "tiny_v2": [1, 42, 21, 8],
    # vggt_v8, |P| = 171: from one block to every candidate, m_0 from 0 to 30 per head
    "vggt_v8": [8, 43, 2, 120, 171, 1, 17, 64, 5, 99, 3, 150, 33, 10, 77, 25],
    # the same spread with every first swap count at most 17
    "vggt_v8_small_m": [8, 43, 2, 68, 171, 1, 17, 64, 5, 30, 3, 69, 33, 10, 50, 25],
}


def _check_csr_rows(layer, D):
    """Every row of the CSR lists exactly the complement of its drop set (dense query rows:
    every block), with the length its own head's budget gives."""
    rp, ci = layer.csr()
    ns = layer.nb - layer.ncand
    assert rp.size == layer.H * layer.nq + 1 and rp[0] == 0 and rp[-1] == ci.size
    for h in range(layer.H):
        for i in range(layer.nq):
            k = ci[rp[h * layer.nq + i]:rp[h * layer.nq + i + 1]]
            if i >= layer.nqc:
                assert k.tolist() == list(range(layer.nb)), (h, i)
            else:
                assert k.size == layer.c_h[h] + ns, (h, i, k.size)
                assert np.array_equal(k, np.nonzero(~D[h, i])[0]), (h, i)


@pytest.mark.parametrize("budgets,q_block", [("tiny_v2", 64), ("tiny_v2", 128), ("vggt_v8", 64),
                                             ("vggt_v8", 128), ("vggt_v8_small_m", 64),
                                             ("vggt_v8_small_m", 128)])
def test_unequal_head_budgets(budgets, q_block):
    """Per-head budgets c_h that differ across the heads (one block, every candidate, and
    values between): drop sets and drift of every row against the oracle, CSR rows of
    per-head lengths at per-head offsets, and attention on rows of every head."""
    wl = synth.WORKLOADS[budgets.replace("_small_m", "")]
    c_h = UNEQUAL_BUDGETS[budgets]
    assert len(c_h) == wl.heads and max(c_h) == wl.n_candidates and min(c_h) == 1
    layer = G.Layer(synth.make_inputs(wl), wl.n_special, c_h, wl.rounds, wl.rho,
                    q_block=q_block).run()
    sel = layer.oracle_select()
    r = G.compare_selection(layer, sel)
    G.check_selection(r)
    assert r["exact"] >= 0.95 * (r["exact"] + r["near"]), r
    D = layer.drop_sets()
    _check_csr_rows(layer, D)
    J0 = layer.ws("J0", shape=(layer.H, layer.nq))
    Jb = layer.buf.J_best.cpu().numpy().reshape(layer.H, layer.nq)
    assert np.all(Jb[:, :layer.nqc] <= J0[:, :layer.nqc])
    for h, c in enumerate(c_h):  # nothing dropped: J = 0 up to rounding; no swaps: J0 kept
        if c == layer.ncand:
            assert np.all(Jb[h, :layer.nqc] <= 1e-9 * Jb.max())
        if all(m <= 0 for m in [min(x, c, layer.ncand - c) for x in O.swap_schedule(c, wl.rounds, wl.rho)]):
            assert np.array_equal(Jb[h, :layer.nqc], J0[h, :layer.nqc])
    rng = np.random.default_rng(4)
    rows = []
    for h in range(layer.H):
        rows += [(h, int(i)) for i in rng.choice(layer.nqc, min(3, layer.nqc), replace=False)]
        rows.append((h, layer.nq - 1))
    a = G.compare_attention(layer, rows)
    assert a["max_abs"] <= G.ATT_MAX_ABS and a["mean_rel"] <= G.ATT_MEAN_REL, a


@pytest.mark.parametrize("q_block", [64, 128])
def test_unequal_head_budgets_edge_shape(q_block):
    """Three heads with budgets 1, |P| and 4 on a ragged sequence with special tokens."""
    N, H, ns, R = 64 * 10 + 17, 3, 5, 3
    inp = synth.make_random_layer(N, H, 64 * H, seed=N + 31)
    nc = O.n_candidates(N, ns)
    c_h = [1, nc, 4]
    layer = G.Layer(inp, ns, c_h, R, q_block=q_block).run()
    r = G.compare_selection(layer, layer.oracle_select())
    G.check_selection(r)
    _check_csr_rows(layer, layer.drop_sets())
    a = G.compare_attention(layer, [(h, i) for h in range(H) for i in range(layer.nq)])
    assert a["max_abs"] <= G.ATT_MAX_ABS and a["mean_rel"] <= G.ATT_MEAN_REL, a


# ---------------------------------------------------------------------------------------
# The headline layer on every row
# ---------------------------------------------------------------------------------------
def test_headline_shape_every_row():
    """32 views, 16 heads, 90% sparsity, R = 3: the drop set and drift of every one of the
    10,944 candidate rows against the oracle (run on every host core in spawned processes),
    and attention on 500 rows: every dense query row (the special-token blocks of every
    head) and a seeded sample of the sparse ones."""
    import time
    import oracle_pool
    layer, wl = layer_for("vggt_v32")
    layer.run()
    rows = [(h, i) for h in range(layer.H) for i in range(layer.nq)]
    t0 = time.perf_counter()
    sel = oracle_pool.select_rows(layer.pooled(), layer.W_o(), layer.c_h, layer.rounds, layer.rho,
                                  rows)
    t_oracle = time.perf_counter() - t0
    assert len(sel) == len(rows)
    r = G.compare_selection(layer, sel)
    print(f"oracle {t_oracle:.1f} s", r)
    G.check_selection(r)
    assert r["exact"] + r["near"] == layer.H * layer.nqc == 10944
    assert r["exact"] >= 0.95 * (r["exact"] + r["near"]), r
    D = layer.drop_sets()
    _check_csr_rows(layer, D)
    dense = [(h, i) for h in range(layer.H) for i in range(layer.nqc, layer.nq)]
    sparse = [(h, i) for h in range(layer.H) for i in range(layer.nqc)]
    rng = np.random.default_rng(9)
    pick = rng.choice(len(sparse), 500 - len(dense), replace=False)
    arows = dense + [sparse[k] for k in sorted(pick)]
    assert len(arows) == 500 and len(dense) == 48
    a = G.compare_attention(layer, arows)
    print(a)
    assert a["max_abs"] <= G.ATT_MAX_ABS and a["mean_rel"] <= G.ATT_MEAN_REL, a
