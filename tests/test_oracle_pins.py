"""Pins of the fp64 oracle against what the paper and mathematics fix.

Each test checks the oracle against an independent statement: np.roll for the
shifted partition (Sec. 2.2 window shift), pair enumeration for pooled affinity
(Eq. for q_b/k_b and S = q_b k_b^T), subset search for Top-k gating, a textbook
numpy softmax for the attention (rho = 0 and masked), closed forms for the
sparsity rule (Algorithm 1, k = floor(Tb*rho)). A plausible mistake in the oracle
(a wrong shift sign, a transposed S, a kept/dropped swap, a missing scale, a
wrong normaliser) fails at least one of them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_geometry.json")


# ----------------------------------------------------------------------------- helpers
def roll_partition(H, W, blk, shift):
    """Literal torch.roll semantics: roll the token-index grid, cut 8x8 tiles."""
    grid = np.arange(H * W).reshape(H, W)
    rolled = np.roll(grid, shift=(shift[0], shift[1]), axis=(0, 1))
    lab = np.empty(H * W, dtype=np.int64)
    bw = W // blk
    for br in range(H // blk):
        for bc in range(bw):
            tile = rolled[br * blk:(br + 1) * blk, bc * blk:(bc + 1) * blk]
            lab[tile.ravel()] = br * bw + bc
    return lab


def numpy_masked_softmax_attention(Q, K, V, allowed, scale):
    """Textbook softmax(scale * Q K^T) V with -inf outside ``allowed`` (fp64)."""
    a = scale * (Q @ K.T)
    a = np.where(allowed, a, -np.inf)
    mx = a.max(axis=1, keepdims=True)
    e = np.exp(a - mx)
    s = e.sum(axis=1, keepdims=True)
    P = e / s
    return P @ V, (mx + np.log(s))[:, 0], P


def expand_mask(labels, idx):
    """M(n, m) = 1 iff label(m) is kept for label(n) (Algorithm 1 ExpandMask)."""
    N = labels.shape[0]
    Tb = idx.shape[0]
    G = np.zeros((Tb, Tb), dtype=bool)
    for i in range(Tb):
        G[i, idx[i]] = True
    return G[labels[:, None], labels[None, :]]


# ----------------------------------------------------------------------------- a1 partition
@pytest.mark.parametrize("H,W", [(16, 16), (32, 32), (16, 40), (64, 64)])
@pytest.mark.parametrize("shift", [(0, 0), (4, 4), (-4, -4), (3, -5), (8, 0), (-1, 12), (4, 0)])
def test_partition_matches_literal_roll(H, W, shift):
    got = oracle.partition(H, W, 8, shift)
    want = roll_partition(H, W, 8, shift)
    assert np.array_equal(got, want)


@pytest.mark.parametrize("shift", [(0, 0), (4, 4), (-4, -4), (2, 6)])
def test_partition_invariants(shift):
    H, W = 32, 48
    lab = oracle.partition(H, W, 8, shift)
    Tb = H * W // 64
    counts = np.bincount(lab, minlength=Tb)
    assert counts.shape[0] == Tb and np.all(counts == 64)  # every token once, 64 per block
    for b in range(Tb):  # each block is an 8x8 cyclically contiguous window
        toks = np.nonzero(lab == b)[0]
        rows = sorted(set((toks // W).tolist()))
        cols = sorted(set((toks % W).tolist()))
        assert len(rows) == 8 and len(cols) == 8
        r0 = [r for r in rows if (r - 1) % H not in rows]
        c0 = [c for c in cols if (c - 1) % W not in cols]
        assert len(r0) == 1 and len(c0) == 1
        assert set(rows) == {(r0[0] + t) % H for t in range(8)}
        assert set(cols) == {(c0[0] + t) % W for t in range(8)}


def test_plus_minus_four_give_the_same_windows():
    """Delta=(4,4) and (-4,-4) on an 8-periodic grid give the same set of windows."""
    H, W = 64, 64
    a = oracle.partition(H, W, 8, (4, 4))
    b = oracle.partition(H, W, 8, (-4, -4))
    sets_a = {frozenset(np.nonzero(a == i)[0].tolist()) for i in range(64)}
    sets_b = {frozenset(np.nonzero(b == i)[0].tolist()) for i in range(64)}
    assert sets_a == sets_b
    # and they differ from the unshifted windows
    c = oracle.partition(H, W, 8, (0, 0))
    sets_c = {frozenset(np.nonzero(c == i)[0].tolist()) for i in range(64)}
    assert sets_a != sets_c


# ----------------------------------------------------------------------------- a2/a3 pooling + affinity
@pytest.mark.parametrize("shift", [(0, 0), (4, 4), (-3, 5)])
def test_affinity_equals_pair_enumeration(shift):
    """S_ij = (1/64^2) sum_{n in i} sum_{m in j} <q_n, k_m>, by explicit pair loops."""
    rng = np.random.default_rng(1)
    H = W = 16
    d = 8
    N = H * W
    Q = rng.standard_normal((N, d))
    K = rng.standard_normal((N, d))
    lab = roll_partition(H, W, 8, shift)
    Tb = 4
    want = np.zeros((Tb, Tb))
    for n in range(N):
        for m in range(N):
            want[lab[n], lab[m]] += float(np.dot(Q[n], K[m]))
    want /= 64.0 * 64.0
    olab = oracle.partition(H, W, 8, shift)
    S = oracle.affinity(oracle.pool(Q, olab, Tb), oracle.pool(K, olab, Tb))
    np.testing.assert_allclose(S, want, rtol=1e-12, atol=1e-12)


def test_pool_constant_blocks_closed_form():
    H = W = 16
    lab = oracle.partition(H, W, 8, (4, 4))
    rng = np.random.default_rng(2)
    means = rng.standard_normal((4, 5))
    X = means[lab]
    np.testing.assert_allclose(oracle.pool(X, lab, 4), means, rtol=1e-14, atol=1e-15)


def test_affinity_is_not_transposed():
    qb = np.array([[1.0, 0.0], [0.0, 2.0]])
    kb = np.array([[3.0, 5.0], [7.0, 11.0]])
    S = oracle.affinity(qb, kb)
    assert S.tolist() == [[3.0, 7.0], [10.0, 22.0]]  # S[i][j] = <qb_i, kb_j>


# ----------------------------------------------------------------------------- a4 gate
@pytest.mark.parametrize("Tb", [4, 5, 6, 8])
def test_gate_keeps_max_sum_subset(Tb):
    """With distinct values, the kept set is the unique size-keep subset of max sum."""
    rng = np.random.default_rng(Tb)
    S = rng.standard_normal((Tb, Tb))
    for k_drop in range(Tb):
        keep = Tb - k_drop
        got = oracle.gate(S, k_drop)
        for i in range(Tb):
            best = max(itertools.combinations(range(Tb), keep), key=lambda c: S[i, list(c)].sum())
            assert got[i].tolist() == list(best)


def test_gate_direction_and_ties():
    Tb = 8
    up = np.tile(np.arange(Tb, dtype=float), (Tb, 1))
    assert oracle.gate(up, 5).tolist() == [[5, 6, 7]] * Tb  # largest kept
    assert oracle.gate(-up, 5).tolist() == [[0, 1, 2]] * Tb  # smallest dropped
    flat = np.zeros((Tb, Tb))
    assert oracle.gate(flat, 6).tolist() == [[0, 1]] * Tb  # ties keep the lower label
    # a tie at the boundary only: values 3,1,1,0 -> keep 2 -> {0, 1}
    S = np.array([[3.0, 1.0, 1.0, 0.0]] * 4)
    assert oracle.gate(S, 2).tolist() == [[0, 1]] * 4
    # -0.0 and +0.0 are equal values: the lower label is kept
    S = np.array([[-0.0, 0.0, -1.0, -2.0]] * 4)
    assert oracle.gate(S, 3).tolist() == [[0]] * 4


def test_gate_invariants_random():
    rng = np.random.default_rng(5)
    Tb = 64
    S = rng.standard_normal((Tb, Tb))
    for k_drop in (0, 1, 32, 53, 63):
        idx = oracle.gate(S, k_drop)
        assert idx.shape == (Tb, Tb - k_drop)
        for i in range(Tb):
            row = idx[i]
            assert np.all(np.diff(row) > 0) and row.min() >= 0 and row.max() < Tb
            dropped = np.setdiff1d(np.arange(Tb), row)
            if len(dropped):
                assert S[i, row].min() >= S[i, dropped].max()


# ----------------------------------------------------------------------------- sparsity rule
def test_sparsity_rule_closed_forms():
    g = json.load(open(GOLDEN))
    assert g["vae_example"]["tokens"] == (g["vae_example"]["image_px"] // 8 // 2) ** 2
    Tb512 = g["vae_example"]["tokens"] // g["block"]["tokens_per_block"]
    assert Tb512 == 16
    # Algorithm 1: k = floor(Tb * rho) dropped
    cases = [(16, 0.75, 12), (16, 0.8416, 13), (64, 0.8416, 53), (64, 0.85, 54),
             (256, 0.84, 215), (256, 0.9, 230), (4, 0.75, 3), (64, 0.0, 0)]
    for Tb, rho, k in cases:
        assert oracle.drop_count(Tb, rho) == k == math.floor(Tb * rho)
        assert oracle.keep_count(Tb, rho) == Tb - k
    # realised sparsity equals rho when Tb*rho is an integer (75% of 16 blocks)
    assert oracle.drop_count(16, g["sparsity"]["vanilla"]) / 16 == g["sparsity"]["vanilla"]


# ----------------------------------------------------------------------------- whole mask, crafted inputs
@pytest.mark.parametrize("shift", [(0, 0), (4, 4)])
@pytest.mark.parametrize("sign", [1.0, -1.0])
def test_build_mask_crafted_block_means(shift, sign):
    """K tokens of block j equal (j+1) e1 and Q tokens equal sign*e1, so S_ij = sign*(j+1)."""
    H = W = 32
    d = 64
    lab = roll_partition(H, W, 8, shift)
    Tb = 16
    K = np.zeros((1, 1, H * W, d))
    K[0, 0, :, 0] = lab + 1.0
    Q = np.zeros((1, 1, H * W, d))
    Q[0, 0, :, 0] = sign
    rho = 0.75
    keep = Tb - math.floor(Tb * rho)
    idx, cnt, S = oracle.build_mask(Q, K, H, W, 8, shift, rho, return_scores=True)
    want_S = sign * np.tile(np.arange(1, Tb + 1, dtype=float), (Tb, 1))
    np.testing.assert_array_equal(S[0, 0], want_S)
    want = list(range(Tb - keep, Tb)) if sign > 0 else list(range(keep))
    assert idx[0, 0].tolist() == [want] * Tb
    assert np.all(cnt == keep)


# ----------------------------------------------------------------------------- a6 attention
@pytest.mark.parametrize("shift", [(0, 0), (4, 4), (-4, -4), (3, 1)])
def test_rho_zero_equals_dense_softmax(shift):
    rng = np.random.default_rng(7)
    H = W = 16
    N, d = H * W, 64
    Q, K, V = (rng.standard_normal((1, 2, N, d)) for _ in range(3))
    idx, cnt = oracle.build_mask(Q, K, H, W, 8, shift, 0.0)
    assert idx.shape[-1] == 4 and np.all(cnt == 4)
    O, lse = oracle.forward(Q, K, V, idx, H, W, 8, shift)
    for h in range(2):
        want_O, want_lse, _ = numpy_masked_softmax_attention(
            Q[0, h], K[0, h], V[0, h], np.ones((N, N), bool), 1 / 8.0)
        np.testing.assert_allclose(O[0, h], want_O, rtol=1e-10, atol=1e-12)
        np.testing.assert_allclose(lse[0, h], want_lse, rtol=1e-12, atol=1e-12)
    Od, lsed = oracle.dense_forward(Q, K, V)
    np.testing.assert_allclose(Od, O, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(lsed, lse, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("shift", [(0, 0), (4, 4), (2, -6)])
def test_masked_attention_equals_numpy_masked_softmax(shift):
    rng = np.random.default_rng(11)
    H, W = 16, 24
    N, d = H * W, 64
    Q, K, V = (rng.standard_normal((1, 1, N, d)) for _ in range(3))
    rho = 0.5
    idx, _ = oracle.build_mask(Q, K, H, W, 8, shift, rho)
    O, lse = oracle.forward(Q, K, V, idx, H, W, 8, shift, scale=0.3)
    allowed = expand_mask(roll_partition(H, W, 8, shift), idx[0, 0])
    want_O, want_lse, P = numpy_masked_softmax_attention(Q[0, 0], K[0, 0], V[0, 0], allowed, 0.3)
    np.testing.assert_allclose(O[0, 0], want_O, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(lse[0, 0], want_lse, rtol=1e-12, atol=1e-12)
    # realised density: each query sees exactly keep*64 keys
    assert np.all(allowed.sum(axis=1) == idx.shape[-1] * 64)
    np.testing.assert_allclose(P.sum(axis=1), 1.0, rtol=0, atol=1e-12)


def test_attention_rows_normalised_and_lse_definition():
    rng = np.random.default_rng(3)
    H = W = 16
    N, d = H * W, 64
    Q, K = (rng.standard_normal((1, 1, N, d)) for _ in range(2))
    ones = np.ones((1, 1, N, d))
    idx, _ = oracle.build_mask(Q, K, H, W, 8, (4, 4), 0.75)
    O, lse = oracle.forward(Q, K, ones, idx, H, W, 8, (4, 4))
    np.testing.assert_allclose(O, 1.0, rtol=0, atol=1e-13)  # sum_m P_nm = 1
    lab = roll_partition(H, W, 8, (4, 4))
    allowed = expand_mask(lab, idx[0, 0])
    a = (Q[0, 0] @ K[0, 0].T) / 8.0
    for n in range(0, N, 17):
        want = math.log(sum(math.exp(x) for x in a[n][allowed[n]]))
        assert abs(lse[0, 0, n] - want) < 1e-12


def test_keep_one_own_block_is_local_attention():
    rng = np.random.default_rng(4)
    H = W = 16
    N, d = H * W, 64
    Q, K, V = (rng.standard_normal((N, d)) for _ in range(3))
    lab = oracle.partition(H, W, 8, (4, 4))
    idx = np.arange(4, dtype=np.int32)[:, None]  # each block attends only to itself
    O, lse = oracle.attention(Q, K, V, lab, idx)
    for b in range(4):
        toks = np.nonzero(roll_partition(H, W, 8, (4, 4)) == b)[0]
        want_O, want_lse, _ = numpy_masked_softmax_attention(
            Q[toks], K[toks], V[toks], np.ones((64, 64), bool), 1 / 8.0)
        np.testing.assert_allclose(O[toks], want_O, rtol=1e-10, atol=1e-12)
        np.testing.assert_allclose(lse[toks], want_lse, rtol=1e-12, atol=1e-12)


def test_oracle_rejects_bad_arguments():
    with pytest.raises(ValueError):
        oracle.partition(12, 16, 8, (0, 0))  # 12 is not a multiple of 8
    with pytest.raises(ValueError):
        oracle.gate(np.zeros((4, 4)), 4)  # keep would be 0


def test_attention_rows_matches_numpy_on_sampled_rows():
    rng = np.random.default_rng(12)
    H, W = 16, 32
    N, d = H * W, 64
    Q, K, V = (rng.standard_normal((N, d)) for _ in range(3))
    lab = oracle.partition(H, W, 8, (4, 4))
    idx = oracle.gate(rng.standard_normal((8, 8)), 5)
    rows = np.array([0, 5, 77, 300, N - 1], dtype=np.int32)
    O, lse = oracle.attention_rows(Q, K, V, lab, idx, rows)
    allowed = expand_mask(roll_partition(H, W, 8, (4, 4)), idx)
    want_O, want_lse, _ = numpy_masked_softmax_attention(Q, K, V, allowed, 1 / 8.0)
    np.testing.assert_allclose(O, want_O[rows], rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(lse, want_lse[rows], rtol=1e-12, atol=1e-12)


# ----------------------------------------------------------------------------- text segment
def algorithm1_joint_literal(Qt, Kt, Vt, Q, K, V, block_of, idx, scale):
    """Algorithm 1 written out densely: G from the kept lists, M_img = ExpandMask(G),
    M = Pad(M_img, T_txt, axis=(0, 1)) with ones, Q, K, V = [text; image], masked softmax
    attention over the whole sequence, return the image rows O[T_txt:] (and their lse)."""
    Tt, N = Kt.shape[0], K.shape[0]
    Tb = idx.shape[0]
    G = np.zeros((Tb, Tb), dtype=bool)
    for i in range(Tb):
        G[i, idx[i]] = True
    M_img = G[block_of][:, block_of]
    M = np.ones((Tt + N, Tt + N), dtype=bool)
    M[Tt:, Tt:] = M_img
    Qa, Ka, Va = np.vstack([Qt, Q]), np.vstack([Kt, K]), np.vstack([Vt, V])
    a = scale * (Qa @ Ka.T)
    a = np.where(M, a, -np.inf)
    mx = a.max(axis=1, keepdims=True)
    e = np.exp(a - mx)
    s = e.sum(axis=1, keepdims=True)
    return (e / s @ Va)[Tt:], (mx + np.log(s))[Tt:, 0]


@pytest.mark.parametrize("Tt,shift", [(5, (4, 4)), (13, (0, 0)), (1, (3, -5))])
def test_joint_attention_is_algorithm1_with_padded_mask(Tt, shift):
    rng = np.random.default_rng(40 + Tt)
    H = W = 16
    N, d = H * W, 8
    Q, K, V = (rng.standard_normal((N, d)) for _ in range(3))
    Qt, Kt, Vt = (rng.standard_normal((Tt, d)) for _ in range(3))
    lab = oracle.partition(H, W, 8, shift)
    idx = np.array([[0, 3], [1, 2], [0, 2], [1, 3]], dtype=np.int32)
    O, lse = oracle.attention_joint(Q, K, V, Kt, Vt, lab, idx)
    O_ref, lse_ref = algorithm1_joint_literal(Qt, Kt, Vt, Q, K, V, lab, idx, 1 / np.sqrt(d))
    np.testing.assert_allclose(O, O_ref, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, lse_ref, rtol=0, atol=1e-12)
    # the text queries do not reach the image rows Algorithm 1 returns
    O2, _ = algorithm1_joint_literal(Qt + 3.0, Kt, Vt, Q, K, V, lab, idx, 1 / np.sqrt(d))
    np.testing.assert_allclose(O2, O_ref, rtol=0, atol=0)


def test_joint_attention_reductions():
    rng = np.random.default_rng(7)
    H = W = 16
    N, d, Tt = H * W, 8, 9
    Q, K, V = (rng.standard_normal((N, d)) for _ in range(3))
    Kt, Vt = (rng.standard_normal((Tt, d)) for _ in range(2))
    lab = oracle.partition(H, W, 8, (4, 4))
    idx = np.array([[1, 2], [0, 3], [2, 3], [0, 1]], dtype=np.int32)
    # no text tokens: the image-only attention
    O0, l0 = oracle.attention_joint(Q, K, V, Kt[:0], Vt[:0], lab, idx)
    Oi, li = oracle.attention(Q, K, V, lab, idx)
    np.testing.assert_array_equal(O0, Oi)
    np.testing.assert_array_equal(l0, li)
    # every image block kept: dense softmax over the concatenated keys [text; image]
    full = np.tile(np.arange(4, dtype=np.int32), (4, 1))
    Of, lf = oracle.attention_joint(Q, K, V, Kt, Vt, lab, full)
    Od, ld, _ = numpy_masked_softmax_attention(Q, np.vstack([Kt, K]), np.vstack([Vt, V]),
                                               np.ones((N, Tt + N), dtype=bool), 1 / np.sqrt(d))
    np.testing.assert_allclose(Of, Od, atol=1e-12)
    np.testing.assert_allclose(lf, ld, atol=1e-12)
    # constant values: every output row is that constant (the weights sum to one)
    c = rng.standard_normal(d)
    Oc, _ = oracle.attention_joint(Q, K, np.tile(c, (N, 1)), Kt, np.tile(c, (Tt, 1)), lab, idx)
    np.testing.assert_allclose(Oc, np.tile(c, (N, 1)), atol=1e-13)
    # a text key far above every image score takes all the weight: O = its value
    Kt2 = Kt.copy()
    Q2 = np.tile(rng.standard_normal(d), (N, 1))
    Kt2[4] = 40.0 * Q2[0]
    Oh, _ = oracle.attention_joint(Q2, K, V, Kt2, Vt, lab, idx)
    np.testing.assert_allclose(Oh, np.tile(Vt[4], (N, 1)), atol=1e-9)


# ----------------------------------------------------------------------------- backward
def numpy_masked_attention_backward(Q, K, V, G, allowed, scale):
    """Textbook matrix-form gradients of O = softmax(scale Q K^T, masked) V for dL/dO = G:
    dV = P^T G, dP = G V^T, dS = P * (dP - rowsum(dP * P)), dQ = scale dS K, dK = scale dS^T Q."""
    _, _, P = numpy_masked_softmax_attention(Q, K, V, allowed, scale)
    dV = P.T @ G
    dP = G @ V.T
    dS = P * (dP - (dP * P).sum(axis=1, keepdims=True))
    return scale * dS @ K, scale * dS.T @ Q, dV


def _bwd_case(shift, seed):
    rng = np.random.default_rng(seed)
    H = W = 16
    N, d = H * W, 8
    Q, K, V, G = (rng.standard_normal((N, d)) for _ in range(4))
    lab = oracle.partition(H, W, 8, shift)
    idx = np.array([[0, 3], [1, 2], [0, 2], [1, 3]], dtype=np.int32)
    return Q, K, V, G, lab, idx, d


@pytest.mark.parametrize("shift", [(4, 4), (0, 0), (3, -5)])
def test_backward_equals_matrix_form_of_masked_softmax(shift):
    Q, K, V, G, lab, idx, d = _bwd_case(shift, 60)
    allowed = np.zeros((Q.shape[0], Q.shape[0]), dtype=bool)
    for n in range(Q.shape[0]):
        allowed[n, np.isin(lab, idx[lab[n]])] = True
    dQ, dK, dV = oracle.attention_backward(Q, K, V, G, lab, idx)
    rQ, rK, rV = numpy_masked_attention_backward(Q, K, V, G, allowed, 1 / np.sqrt(d))
    for a, b in ((dQ, rQ), (dK, rK), (dV, rV)):
        np.testing.assert_allclose(a, b, rtol=0, atol=1e-12)


def test_backward_matches_central_finite_differences():
    """dL/dX for L = sum(G * O(Q, K, V)), at sampled entries, by central differences of the
    forward oracle (h = 1e-5: truncation and rounding errors far below 1e-7)."""
    Q, K, V, G, lab, idx, d = _bwd_case((4, 4), 61)
    dQ, dK, dV = oracle.attention_backward(Q, K, V, G, lab, idx)

    def loss(Qx, Kx, Vx):
        O, _ = oracle.attention(Qx, Kx, Vx, lab, idx)
        return float((G * O).sum())

    rng = np.random.default_rng(62)
    h = 1e-5
    for which, grad in ((0, dQ), (1, dK), (2, dV)):
        for _ in range(12):
            n, c = int(rng.integers(Q.shape[0])), int(rng.integers(d))
            args = [Q.copy(), K.copy(), V.copy()]
            args[which][n, c] += h
            lp = loss(*args)
            args[which][n, c] -= 2 * h
            lm = loss(*args)
            assert abs((lp - lm) / (2 * h) - grad[n, c]) < 1e-7, (which, n, c)


def test_backward_key_gradients_sum_to_zero():
    """Each query row's ds sums to zero (sum_m p (dp - D) = D - D), so sum_m dK_m = 0; a
    sign or normaliser error breaks it. dV sums to the column sums of dO (rows of P sum to 1)."""
    Q, K, V, G, lab, idx, d = _bwd_case((4, 4), 63)
    _, dK, dV = oracle.attention_backward(Q, K, V, G, lab, idx)
    np.testing.assert_allclose(dK.sum(axis=0), 0.0, atol=1e-12)
    np.testing.assert_allclose(dV.sum(axis=0), G.sum(axis=0), atol=1e-11)


# ----------------------------------------------------------------------------- Haar wavelets
def test_haar_hand_example_and_reconstruction():
    """A 2 x 2 window by hand, perfect reconstruction (the bank is orthonormal), energy
    preservation, and a constant image that has only an LL band."""
    x = np.array([[[1.0, 2.0], [3.0, 5.0]]])  # a=1 b=2 c=3 d=5
    y = oracle.haar_dwt(x)
    np.testing.assert_allclose(y[:, 0, 0], [11 / 2, -3 / 2, -5 / 2, 1 / 2])  # LL HL LH HH
    rng = np.random.default_rng(70)
    x = rng.standard_normal((3, 6, 8))
    y = oracle.haar_dwt(x)
    np.testing.assert_allclose(oracle.haar_iwt(y, 3), x, atol=1e-14)
    np.testing.assert_allclose((y ** 2).sum(), (x ** 2).sum(), rtol=1e-13)
    yc = oracle.haar_dwt(np.full((2, 4, 4), 3.0))
    np.testing.assert_allclose(yc[:2], 6.0)
    np.testing.assert_allclose(yc[2:], 0.0)


def test_haar_bands_are_separable_1d_haar():
    """The 2-D bands equal the 1-D orthonormal Haar (sum, difference over sqrt 2) along
    the width, then along the height: LL = low-low, HL = width-high/height-low, ..."""
    rng = np.random.default_rng(71)
    x = rng.standard_normal((2, 8, 6))
    s2 = np.sqrt(2.0)
    lo_w = (x[..., 0::2] + x[..., 1::2]) / s2
    hi_w = (x[..., 0::2] - x[..., 1::2]) / s2
    bands = [(lo_w[..., 0::2, :] + lo_w[..., 1::2, :]) / s2, (hi_w[..., 0::2, :] + hi_w[..., 1::2, :]) / s2,
             (lo_w[..., 0::2, :] - lo_w[..., 1::2, :]) / s2, (hi_w[..., 0::2, :] - hi_w[..., 1::2, :]) / s2]
    y = oracle.haar_dwt(x)
    for s, b in enumerate(bands):
        np.testing.assert_allclose(y[s * 2:(s + 1) * 2], b, atol=1e-14)
    # dropping HH: the inverse of the three kept bands is x minus the HH contribution
    y3 = oracle.haar_dwt(x, nb=3)
    np.testing.assert_array_equal(y3, y[:6])
    np.testing.assert_allclose(oracle.haar_iwt(y3, 2, nb=3) + oracle.haar_iwt(
        np.concatenate([np.zeros_like(y[:6]), y[6:]]), 2), x, atol=1e-14)


def test_haar_pyramid_closed_forms():
    """Level L of the pyramid: LL is the sum over each 2^L x 2^L tile divided by 2^L (each
    orthonormal level doubles a constant); energy splits exactly over LL_L and the detail bands
    of every level; a constant image has no detail at any level."""
    rng = np.random.default_rng(72)
    x = rng.standard_normal((2, 3, 16, 24))
    L = 3
    ys = oracle.haar_dwt_pyramid(x, L)
    assert [y.shape for y in ys] == [(2, 12, 8, 12), (2, 12, 4, 6), (2, 12, 2, 3)]
    tile = x.reshape(2, 3, 2, 8, 3, 8).sum(axis=(3, 5)) / 2 ** L
    np.testing.assert_allclose(ys[-1][:, :3], tile, atol=1e-13)
    energy = (ys[-1][:, :3] ** 2).sum() + sum((y[:, 3:] ** 2).sum() for y in ys)
    np.testing.assert_allclose(energy, (x ** 2).sum(), rtol=1e-13)
    yc = oracle.haar_dwt_pyramid(np.full((1, 2, 8, 8), -1.5), 3)
    for y in yc:
        np.testing.assert_allclose(y[:, 2:], 0.0, atol=1e-15)
    np.testing.assert_allclose(yc[-1][:, :2], -1.5 * 8, atol=1e-14)


def test_haar_pyramid_inverse_reads_only_deepest_ll_and_details():
    """The inverse pyramid gives x back, and the LL bands of the shallower levels (which the
    decoder recomputes) do not enter it; with nb = 3 it loses exactly the HH bands."""
    rng = np.random.default_rng(73)
    x = rng.standard_normal((2, 4, 16, 8))
    ys = oracle.haar_dwt_pyramid(x, 3)
    np.testing.assert_allclose(oracle.haar_iwt_pyramid(ys, 4), x, atol=1e-13)
    spoiled = [y.copy() for y in ys]
    for y in spoiled[:-1]:
        y[:, :4] = 1e6
    np.testing.assert_allclose(oracle.haar_iwt_pyramid(spoiled, 4), x, atol=1e-13)
    y3 = oracle.haar_dwt_pyramid(x, 2, nb=3)
    np.testing.assert_array_equal(y3[0], ys[0][:, :12])
    # HH removed at both levels: the inverse equals the full inverse with those bands zeroed
    zeroed = [ys[0].copy(), ys[1].copy()]
    zeroed[0][:, 12:] = 0.0
    zeroed[1][:, 12:] = 0.0
    np.testing.assert_allclose(oracle.haar_iwt_pyramid(y3, 4, nb=3), oracle.haar_iwt_pyramid(zeroed, 4),
                               atol=1e-13)


# ----------------------------------------------------------------------------- RoPE + QKV
def test_rope_hand_values_and_axes():
    """theta_0 = 1 rad: a unit vector on dimension 0 at row 1 turns to (cos 1, sin 1); on
    dimension 32 at column 2 to (cos 2, sin 2); dimension 2 turns by 10000^(-1/16) per row;
    a row displacement leaves the column half alone and vice versa; token (0, 0) is unchanged."""
    H, W, d = 3, 4, 64
    x = np.zeros((H * W, d))
    x[:, 0] = 1.0
    x[:, 2] = 1.0
    x[:, 32] = 1.0
    y = oracle.rope_2d(x, H, W)
    t = 1 * W + 0  # row 1, column 0
    np.testing.assert_allclose(y[t, :2], [np.cos(1.0), np.sin(1.0)], atol=1e-15)
    th1 = 10000.0 ** (-1 / 16)
    np.testing.assert_allclose(y[t, 2:4], [np.cos(th1), np.sin(th1)], atol=1e-15)
    np.testing.assert_allclose(y[t, 32:34], [1.0, 0.0], atol=1e-15)  # column 0: no turn
    t = 0 * W + 2  # row 0, column 2
    np.testing.assert_allclose(y[t, 32:34], [np.cos(2.0), np.sin(2.0)], atol=1e-15)
    np.testing.assert_allclose(y[t, :4], [1.0, 0.0, 1.0, 0.0], atol=1e-15)
    np.testing.assert_array_equal(y[0], x[0])


def test_rope_is_a_rotation_with_relative_positions():
    """Norms are kept pair by pair, and <R q(p1), R k(p2)> depends only on p1 - p2 on each axis."""
    rng = np.random.default_rng(80)
    H, W, d = 6, 7, 64
    q, k = rng.standard_normal(d), rng.standard_normal(d)
    Rq = oracle.rope_2d(np.tile(q, (H * W, 1)), H, W)
    Rk = oracle.rope_2d(np.tile(k, (H * W, 1)), H, W)
    np.testing.assert_allclose((Rq.reshape(-1, 32, 2) ** 2).sum(-1), np.tile((q.reshape(32, 2) ** 2).sum(-1), (H * W, 1)),
                               rtol=1e-13)
    tok = lambda r, c: r * W + c
    for (r1, c1), (r2, c2), (dr, dc) in (((1, 2), (0, 0), (2, 3)), ((4, 1), (2, 5), (1, 1)), ((0, 6), (3, 0), (2, 0))):
        a = Rq[tok(r1, c1)] @ Rk[tok(r2, c2)]
        b = Rq[tok(r1 + dr, c1 + dc)] @ Rk[tok(r2 + dr, c2 + dc)]
        np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-12)
    # and does change with the offset
    assert abs(Rq[tok(1, 2)] @ Rk[tok(0, 0)] - Rq[tok(1, 3)] @ Rk[tok(0, 0)]) > 1e-6


def test_qkv_projection_layout_and_bias():
    """With Wqkv = [I; 2I; 3I] the projection is X, 2X, 3X cut into heads of 64 consecutive
    channels (Q rows first, then K, then V); the bias is added once; RoPE turns Q and K only."""
    rng = np.random.default_rng(81)
    B, H, W, heads, d = 2, 4, 4, 3, 64
    Dm = heads * d
    X = rng.standard_normal((B, H * W, Dm))
    Wqkv = np.concatenate([np.eye(Dm), 2 * np.eye(Dm), 3 * np.eye(Dm)])
    Q, K, V = oracle.qkv_rope(X, Wqkv, None, heads, H, W)
    heads_of = lambda Y: Y.reshape(B, H * W, heads, d).transpose(0, 2, 1, 3)
    np.testing.assert_allclose(Q, oracle.rope_2d(heads_of(X), H, W), atol=1e-14)
    np.testing.assert_allclose(K, oracle.rope_2d(heads_of(2 * X), H, W), atol=1e-14)
    np.testing.assert_allclose(V, heads_of(3 * X), atol=1e-14)
    bias = rng.standard_normal(3 * Dm)
    Q2, K2, V2 = oracle.qkv_rope(X, Wqkv, bias, heads, H, W)
    np.testing.assert_allclose(V2 - V, np.broadcast_to(bias[2 * Dm:].reshape(heads, 1, d), V.shape), atol=1e-14)
    np.testing.assert_allclose(Q2[:, :, 0] - Q[:, :, 0], np.broadcast_to(bias[:Dm].reshape(heads, d), (B, heads, d)),
                               atol=1e-14)  # token (0, 0): RoPE is the identity there


def test_pooled_blocks_matches_pool_of_each_head():
    rng = np.random.default_rng(82)
    X = rng.standard_normal((1, 2, 16 * 16, 64))
    P = oracle.pooled_blocks(X, 16, 16, 8, (4, 4))
    lab = oracle.partition(16, 16, 8, (4, 4))
    for b in range(4):
        np.testing.assert_allclose(P[0, 1, b], X[0, 1][lab == b].mean(axis=0), atol=1e-14)
