"""Pins of the fp64 oracle to things other than itself (no GPU).

Each test fixes the oracle against what the paper and the mathematics fix:
a library routine that computes the same definition (PyTorch's float64
scaled_dot_product_attention with its own causal semantics, numpy's argmax and
slicing), closed forms, invariants, the decomposition of one softmax over
disjoint key sets, and the worked acceptance case of Fig. 1(c).  Inputs come
from the seeded generator (synth).  A planted mistake in the oracle (a dropped
block term, a j < i mask, swapped read depths, a wrong scale or GQA mapping,
an off-by-one in the append count) fails at least one of these.
"""
import math
import os

import numpy as np
import pytest
import torch

import oracle
import synth
from synth import workloads as wl_mod

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def f64(bits):
    return synth.bf16_bits_to_float(bits).astype(np.float64)


def rand_bits(seed, shape, scale=1.0):
    """bf16 bits of seeded N(0,1)*scale values, via the generator."""
    n = int(np.prod(shape))
    D = shape[-1]
    rows = n // D
    blk = synth.normal_block(seed, synth.T_Q, 0, 0, 0, rows, 0, 1, D, 1.0 / scale)
    return blk.reshape(shape)


def sdpa_reference(q, keys, values, P, scale, G):
    """Library evaluation of Eqs. 2-3 for one sequence: queries of block rows
    sit at positions P..P+T-1 after P padding queries, and PyTorch's is_causal
    (position n sees keys 0..n) gives prefix-visible + in-block causal."""
    T, Hq, D = q.shape
    qq = torch.zeros((1, Hq, P + T, D), dtype=torch.float64)
    qq[0, :, P:, :] = torch.from_numpy(q).permute(1, 0, 2)
    kk = torch.from_numpy(keys).permute(1, 0, 2)[None]
    vv = torch.from_numpy(values).permute(1, 0, 2)[None]
    o = torch.nn.functional.scaled_dot_product_attention(qq, kk, vv, is_causal=True, scale=scale,
                                                         enable_gqa=G > 1)
    return o[0, :, P:, :].permute(1, 0, 2).numpy()


CASES = [  # (P, T, Hq, Hkv, D, scale)
    (0, 4, 4, 4, 64, None),
    (1, 1, 2, 2, 64, None),
    (37, 5, 8, 2, 64, None),
    (130, 16, 8, 2, 128, None),
    (64, 8, 4, 1, 32, 1.0),
    (300, 3, 6, 3, 16, 0.7),
]


@pytest.mark.parametrize("P,T,Hq,Hkv,D,scale", CASES)
def test_matches_library_attention(P, T, Hq, Hkv, D, scale):
    """Oracle == float64 SDPA over [K_C ; K_U], [V_C ; V_U] (Eqs. 2-3), GQA included."""
    seed = 1000 + P + 7 * T + Hq
    q = rand_bits(seed, (T, Hq, D))
    kp, vp = rand_bits(seed + 1, (P, Hkv, D)), rand_bits(seed + 2, (P, Hkv, D))
    kb, vb = rand_bits(seed + 3, (T, Hkv, D)), rand_bits(seed + 4, (T, Hkv, D))
    out, lse = oracle.attend_seq(q, kp, vp, kb, vb, scale=scale)
    sc = 1.0 / math.sqrt(D) if scale is None else scale
    ref = sdpa_reference(f64(q), np.concatenate([f64(kp), f64(kb)]),
                         np.concatenate([f64(vp), f64(vb)]), P, sc, Hq // Hkv)
    np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)
    assert np.all(np.isfinite(lse))


def test_block_len_rows_and_lse_closed_form():
    """Rows past block_len are 0 / -inf; with all keys identical, s_j = s for
    every j and lse = s + ln(n), out = mean of the values (closed form)."""
    P, T, Hq, D = 9, 4, 2, 8
    q = rand_bits(5, (T, Hq, D))
    k1 = rand_bits(6, (1, 1, D))
    kp = np.repeat(k1, P, axis=0)
    kb = np.repeat(k1, T, axis=0)
    vp, vb = rand_bits(7, (P, 1, D)), rand_bits(8, (T, 1, D))
    out, lse = oracle.attend_seq(q, kp, vp, kb, vb, block_len=3)
    assert np.all(out[3] == 0) and np.all(np.isneginf(lse[:, 3]))
    allv = np.concatenate([f64(vp), f64(vb)])[:, 0, :]
    for i in range(3):
        n = P + i + 1
        for h in range(Hq):
            s = np.dot(f64(q)[i, h], f64(k1)[0, 0]) / math.sqrt(D)
            assert abs(lse[h, i] - (s + math.log(n))) < 1e-12
            np.testing.assert_allclose(out[i, h], allv[:n].mean(axis=0), atol=1e-13)


def test_single_key_returns_its_value():
    """One prefix key and no block: weight 1, out = v_0 exactly, lse = s_0."""
    D = 64
    q, k, v = rand_bits(11, (1, 1, D)), rand_bits(12, (1, 1, D)), rand_bits(13, (1, 1, D))
    out, lse = oracle.attend_seq(q, k, v, k, v, use_block=False)
    assert np.array_equal(out[0, 0], f64(v)[0, 0])
    assert lse[0, 0] == pytest.approx(float(np.dot(f64(q)[0, 0], f64(k)[0, 0])) / 8.0, abs=1e-14)
    # empty prefix, block row 0 sees only its own key: out = v_blk[0]
    out, lse = oracle.attend_seq(q, k[:0], v[:0], k, v)
    assert np.array_equal(out[0, 0], f64(v)[0, 0])


def test_zero_query_is_mean_of_attended_values():
    """q = 0: every score is 0, weights are uniform, lse = ln(#keys)."""
    P, T, D = 20, 3, 16
    q = np.zeros((T, 2, D), dtype=np.uint16)
    kp, vp = rand_bits(21, (P, 1, D)), rand_bits(22, (P, 1, D))
    kb, vb = rand_bits(23, (T, 1, D)), rand_bits(24, (T, 1, D))
    out, lse = oracle.attend_seq(q, kp, vp, kb, vb)
    allv = np.concatenate([f64(vp), f64(vb)])[:, 0, :]
    for i in range(T):
        np.testing.assert_allclose(out[i, 0], allv[:P + i + 1].mean(axis=0), atol=1e-13)
        assert lse[0, i] == pytest.approx(math.log(P + i + 1), abs=1e-14)


def test_convex_hull_and_prefix_permutation():
    """Out lies in the per-dim hull of the attended values; permuting prefix
    positions (K and V together) leaves out and lse unchanged."""
    P, T, Hq, Hkv, D = 50, 6, 4, 2, 32
    q = rand_bits(31, (T, Hq, D), scale=3.0)
    kp, vp = rand_bits(32, (P, Hkv, D)), rand_bits(33, (P, Hkv, D))
    kb, vb = rand_bits(34, (T, Hkv, D)), rand_bits(35, (T, Hkv, D))
    out, lse = oracle.attend_seq(q, kp, vp, kb, vb)
    allv = np.concatenate([f64(vp), f64(vb)])
    for i in range(T):
        for h in range(Hq):
            vals = allv[:P + i + 1, h // 2, :]
            assert np.all(out[i, h] <= vals.max(axis=0) + 1e-12)
            assert np.all(out[i, h] >= vals.min(axis=0) - 1e-12)
    perm = np.random.default_rng(0).permutation(P)
    out2, lse2 = oracle.attend_seq(q, kp[perm], vp[perm], kb, vb)
    np.testing.assert_allclose(out2, out, atol=1e-13)
    np.testing.assert_allclose(lse2, lse, atol=1e-13)


def test_disjoint_key_sets_merge_to_one_softmax():
    """Eq. 2 is one softmax over C and U: partial results over disjoint
    prefix chunks (and the block) combine as exp(lse_s - lse) O_s with
    lse = log sum exp(lse_s) into the single-softmax result."""
    P, T, Hq, Hkv, D = 333, 8, 8, 2, 64
    q = rand_bits(41, (T, Hq, D), scale=2.0)
    kp, vp = rand_bits(42, (P, Hkv, D)), rand_bits(43, (P, Hkv, D))
    kb, vb = rand_bits(44, (T, Hkv, D)), rand_bits(45, (T, Hkv, D))
    full_o, full_l = oracle.attend_seq(q, kp, vp, kb, vb)
    cuts = [0, 1, 64, 65, 200, 333]
    parts = [oracle.attend_seq(q, kp, vp, kb, vb, prefix_range=(a, b), use_block=False)
             for a, b in zip(cuts[:-1], cuts[1:])]
    parts.append(oracle.attend_seq(q, kp, vp, kb, vb, prefix_range=(0, 0), use_block=True))
    L = np.stack([p[1] for p in parts])              # [S][Hq][T]
    M = L.max(axis=0)
    lse = M + np.log(np.exp(L - M).sum(axis=0))
    out = sum(np.exp(p[1] - lse).T[:, :, None] * p[0] for p in parts)
    np.testing.assert_allclose(lse, full_l, atol=1e-12)
    np.testing.assert_allclose(out, full_o, atol=1e-12)


def test_mpmath_brute_force_tiny():
    """50-digit evaluation on a tiny case bounds the oracle's rounding."""
    mp = pytest.importorskip("mpmath")
    mp.mp.dps = 50
    P, T, D = 5, 3, 4
    q = rand_bits(51, (T, 1, D), scale=4.0)
    kp, vp = rand_bits(52, (P, 1, D)), rand_bits(53, (P, 1, D))
    kb, vb = rand_bits(54, (T, 1, D)), rand_bits(55, (T, 1, D))
    out, lse = oracle.attend_seq(q, kp, vp, kb, vb, scale=0.9)
    keys = np.concatenate([f64(kp), f64(kb)])[:, 0]
    vals = np.concatenate([f64(vp), f64(vb)])[:, 0]
    for i in range(T):
        n = P + i + 1
        s = [mp.mpf(0.9) * mp.fsum(mp.mpf(float(a)) * mp.mpf(float(b))
                                   for a, b in zip(f64(q)[i, 0], keys[j])) for j in range(n)]
        Z = mp.fsum(mp.e ** x for x in s)
        assert abs(float(mp.log(Z)) - lse[0, i]) < 1e-13
        for d in range(D):
            o = mp.fsum(mp.e ** x * mp.mpf(float(vals[j, d])) for j, x in enumerate(s)) / Z
            assert abs(float(o) - out[i, 0, d]) < 1e-13


def test_whole_cache_reads_key_and_value_depths():
    """The whole-cache oracle reads keys at depth kappa and values at depth nu
    (Eq. 4): it equals the library attention over those two slabs, for
    Mature-V (r, R), Aligned (r, r), Deep K (R, r) and Deep K/V (R, R)."""
    wl = wl_mod.WORKLOADS["tiny"].replace(prefix=(40, 40), block=(3,), batch=2, layers=2)
    R, r = wl.depths, wl.key_depth
    K, V = wl_mod.gen_cache(wl, depths=[r, R])
    q = wl_mod.gen_q(wl, 1)
    kb, vb = wl_mod.gen_block_kv(wl, 1)
    pl, bl = wl.prefix_lens(), wl.block_lens()
    for kap, nu in [(r, R), (r, r), (R, r), (R, R)]:
        out, lse = oracle.attention(K, V, 1, kap, nu, pl, bl, q, kb, vb)
        for b in range(wl.batch):
            P = pl[b]
            ref = sdpa_reference(f64(q[b]), np.concatenate([f64(K[kap - 1, 1, b, :P]), f64(kb[b])]),
                                 np.concatenate([f64(V[nu - 1, 1, b, :P]), f64(vb[b])]), P,
                                 1.0 / math.sqrt(wl.head_dim), 1)
            np.testing.assert_allclose(out[b], ref, atol=1e-12)
    # the two depths really differ in this data, so the depth choice matters
    o1, _ = oracle.attention(K, V, 1, r, R, pl, bl, q, kb, vb)
    o2, _ = oracle.attention(K, V, 1, R, r, pl, bl, q, kb, vb)
    assert np.abs(o1 - o2).max() > 1e-3


def test_invalid_arguments_rejected():
    K = np.zeros((2, 1, 1, 4, 1, 8), dtype=np.uint16)
    q = np.zeros((1, 1, 1, 8), dtype=np.uint16)
    kb = np.zeros((1, 1, 1, 8), dtype=np.uint16)
    with pytest.raises(ValueError):
        oracle.attention(K, K, 0, 3, 1, [0], [1], q, kb, kb)  # depth beyond R
    with pytest.raises(ValueError):
        oracle.attention(K, K, 0, 1, 1, [5], [1], q, kb, kb)  # prefix beyond capacity


# ----------------------------- greedy acceptance -----------------------------

def _read_golden(name):
    rows = [l.split() for l in open(os.path.join(GOLDEN, name)) if l.strip() and l[0] != "#"]
    W, Vv = map(int, rows[0])
    draft = np.array([list(map(int, rows[1]))], dtype=np.int32)
    logits = np.array([[list(map(float, r)) for r in rows[2:2 + W]]], dtype=np.float32)
    exp = list(map(int, rows[2 + W][1:]))
    return draft, logits, exp[0], exp[1], exp[2:]


def test_accept_fig1c_worked_case():
    draft, logits, a, nxt, targets = _read_golden("accept_fig1c.txt")
    acc, tid, nx = oracle.greedy_accept(logits, draft)
    assert acc[0] == a and nx[0] == nxt and list(tid[0]) == targets


def test_accept_edge_cases():
    """All accepted (m = w: no bonus, the last proposal is the next anchor),
    mismatch at the first proposal, mismatch at the last, and ties."""
    rng = np.random.default_rng(3)
    W, Vv = 5, 11
    logits = rng.normal(0, 2, (4, W, Vv)).astype(np.float32)
    am = logits.argmax(axis=2).astype(np.int32)
    draft = am.copy()
    draft[1, 0] = (am[1, 0] + 1) % Vv
    draft[2, W - 1] = (am[2, W - 1] + 1) % Vv
    logits[3, :, :] = 0.0  # all tied: smallest index 0 wins
    draft[3] = [0, 0, 7, 0, 0]
    acc, tid, nx = oracle.greedy_accept(logits, draft)
    assert list(acc) == [W, 0, W - 1, 2]
    assert nx[0] == draft[0, W - 1]
    assert nx[1] == am[1, 0] and nx[2] == am[2, W - 1] and nx[3] == 0
    assert np.array_equal(tid[:3], am[:3]) and np.all(tid[3] == 0)


def test_accept_matches_numpy_argmax_and_planted_lengths():
    """numpy.argmax (first maximum) gives the same targets; the generator's
    planted acceptance lengths come back exactly."""
    a_star, draft, logits = synth.accept_inputs(0, 8, 16, 3000)
    acc, tid, nx = oracle.greedy_accept(logits, draft)
    assert np.array_equal(tid, logits.argmax(axis=2))
    assert np.array_equal(acc, a_star)
    for b in range(8):
        assert nx[b] == (tid[b, acc[b]] if acc[b] < 16 else draft[b, 15])


# ----------------------------------- append ----------------------------------

def test_append_matches_slicing_and_counts():
    """n_b = min(a_b + 1, W) staged positions land at prefix_len[b] at every
    depth and layer; nothing else changes; prefix_len grows by n_b."""
    rng = np.random.default_rng(4)
    R, L, B, cap, H, D, W = 3, 2, 5, 12, 2, 8, 4
    K = rng.integers(0, 65535, (R, L, B, cap, H, D), dtype=np.uint16)
    V = rng.integers(0, 65535, (R, L, B, cap, H, D), dtype=np.uint16)
    kn = rng.integers(0, 65535, (R, L, B, W, H, D), dtype=np.uint16)
    vn = rng.integers(0, 65535, (R, L, B, W, H, D), dtype=np.uint16)
    acc = np.array([0, 1, W - 1, W, 2], dtype=np.int32)
    pl = np.array([0, 3, 8, 7, 0], dtype=np.int32)
    K2, V2, pl2, flag = oracle.kv_append(K, V, kn, vn, acc, pl)
    n = np.array([1, 2, W, W, 3])
    assert flag == 0 and np.array_equal(pl2, pl + n)
    Ke, Ve = K.copy(), V.copy()
    for b in range(B):
        Ke[:, :, b, pl[b]:pl[b] + n[b]] = kn[:, :, b, :n[b]]
        Ve[:, :, b, pl[b]:pl[b] + n[b]] = vn[:, :, b, :n[b]]
    assert np.array_equal(K2, Ke) and np.array_equal(V2, Ve)


def test_append_overflow_leaves_sequence_untouched():
    R, L, B, cap, H, D, W = 2, 1, 2, 6, 1, 8, 4
    K = np.arange(R * L * B * cap * H * D, dtype=np.uint16).reshape(R, L, B, cap, H, D)
    kn = np.full((R, L, B, W, H, D), 7, dtype=np.uint16)
    K2, V2, pl2, flag = oracle.kv_append(K, K, kn, kn, [3, 0], [3, 5])
    assert flag == 1
    assert list(pl2) == [3, 6]                      # seq 0 overflowed, seq 1 fit
    assert np.array_equal(K2[:, :, 0], K[:, :, 0])  # untouched
    assert np.all(K2[:, :, 1, 5] == 7)


# ------------------------------ DAS-Wave readout ------------------------------

def test_wave_widths_eq5():
    """Eq. 5: W_j = min(gamma, W_init + j).  The paper's setting (gamma = 32,
    W_init = 2, J = 24; App. A.2) grows from 2 to 25 and never reaches gamma;
    a small gamma caps the width."""
    assert [oracle.wave_width(32, 2, j) for j in range(24)] == list(range(2, 26))
    assert [oracle.wave_width(8, 2, j) for j in range(10)] == [2, 3, 4, 5, 6, 7, 8, 8, 8, 8]
    assert oracle.wave_width(32, 2, 0) == 2


def test_wave_readout_is_shifted_first_maximum():
    """Eq. 6: the readout of position i becomes the guess of position i + 1
    (numpy.argmax: first maximum); the anchor (position 0) and positions past
    W keep their values; an all-tied row and an all -inf row read out 0."""
    rng = np.random.default_rng(11)
    B, W, Vv, S = 3, 6, 97, 10
    logits = rng.normal(0, 2, (B, W, Vv)).astype(np.float32)
    logits[1, 2, :] = 0.5
    logits[2, 4, :] = -np.inf
    logits[0, 3, [5, 40]] = 50.0  # a planted tie: index 5 wins
    tokens = rng.integers(0, Vv, (B, S)).astype(np.int32)
    out = oracle.wave_readout(logits, tokens)
    exp = tokens.copy()
    exp[:, 1:W + 1] = logits.argmax(axis=2)
    assert np.array_equal(out, exp)
    assert out[0, 4] == 5 and out[1, 3] == 0 and out[2, 5] == 0
    assert np.array_equal(out[:, 0], tokens[:, 0]) and np.array_equal(out[:, W + 1:],
                                                                    tokens[:, W + 1:])


def test_wave_rounds_grow_the_window_with_the_last_readout():
    """Over rounds with W_j from Eq. 5, the candidate that enters the active
    window at round j + 1 (position W_j) is the readout of the last active
    position W_j - 1 at round j (Sec. 3.3); earlier guesses are revised in
    place."""
    rng = np.random.default_rng(12)
    gamma, w_init, J, Vv = 6, 2, 7, 50
    tokens = np.zeros((1, gamma + 1), dtype=np.int32)
    tokens[0, 0] = 9  # anchor x_t
    for j in range(J):
        W = oracle.wave_width(gamma, w_init, j)
        logits = rng.normal(0, 1, (1, W, Vv)).astype(np.float32)
        new = oracle.wave_readout(logits, tokens)
        assert new[0, 0] == 9
        assert new[0, W] == logits[0, W - 1].argmax()  # next candidate enters at W
        tokens = new
    assert oracle.wave_width(gamma, w_init, J - 1) == gamma


# --------------------------- e4m3 storage (variant) ---------------------------

def _torch_e4m3():
    torch = pytest.importorskip("torch")
    if not hasattr(torch, "float8_e4m3fn"):
        pytest.skip("torch without float8_e4m3fn")
    return torch


def test_e4m3_decode_matches_torch_on_every_code():
    torch = _torch_e4m3()
    codes = np.arange(256, dtype=np.uint8)
    ours = oracle.e4m3_decode(codes)
    ref = torch.from_numpy(codes).view(torch.float8_e4m3fn).float().double().numpy()
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan) and nan.sum() == 2   # S.1111.111 only
    assert np.array_equal(ours[~nan], ref[~nan])
    assert ours[0x7E] == 448.0 and ours[0x01] == 2.0 ** -9 and ours[0x08] == 2.0 ** -6


def test_e4m3_encode_round_trip_and_torch_rounding():
    """Every finite code survives decode -> encode; random bf16 values within
    +-448 round like torch's float -> float8_e4m3fn cast (nearest, ties to
    even)."""
    torch = _torch_e4m3()
    codes = np.array([c for c in range(256) if c not in (0x7F, 0xFF)], dtype=np.uint8)
    bits = (oracle.e4m3_decode(codes).astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    assert np.array_equal(oracle.e4m3_from_bf16(bits), codes)
    rng = np.random.default_rng(21)
    x = np.concatenate([rng.normal(0, s, 20000) for s in (1e-3, 0.1, 1.0, 30.0)])
    x = np.clip(x, -448, 448).astype(np.float32)
    b16 = (x.view(np.uint32) >> 16).astype(np.uint16)           # truncate to bf16 values
    xv = (b16.astype(np.uint32) << 16).view(np.float32)
    ref = torch.from_numpy(xv).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(oracle.e4m3_from_bf16(b16), ref)


def test_e4m3_encode_ties_and_saturation():
    def enc(v):
        b = (np.array([v], np.float32).view(np.uint32) >> 16).astype(np.uint16)
        return int(oracle.e4m3_from_bf16(b)[0])
    u = 2.0 ** -9                                   # the subnormal step
    assert [enc(0.5 * u), enc(1.5 * u), enc(2.5 * u), enc(7.5 * u)] == [0x00, 0x02, 0x02, 0x08]
    assert enc(1.0625) == 0x38 and enc(1.1875) == 0x3A   # ties to the even mantissa
    assert [enc(448.0), enc(449.0), enc(464.0), enc(1e30), enc(np.inf)] == [0x7E] * 5
    assert [enc(-449.0), enc(-np.inf)] == [0xFE, 0xFE]
    assert enc(-0.0) == 0x80


def test_e4m3_cache_attention_reduces_to_bf16():
    """With every depth below R holding e4m3-representable bf16 values, the
    e4m3 cache is the same cache: attention_f8 equals attention bit for bit;
    key_depth = value_depth = R reads only the bf16 top."""
    rng = np.random.default_rng(22)
    R, L, B, cap, H, D = 3, 1, 2, 40, 2, 8
    codes = rng.integers(0, 256, (R - 1, L, B, cap, H, D)).astype(np.uint8)
    codes[(codes & 0x7F) == 0x7F] = 0x38            # no NaN
    low_bits = (oracle.e4m3_decode(codes).astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    top = rng.integers(0x3C00, 0x4000, (L, B, cap, H, D)).astype(np.uint16)
    K = np.concatenate([low_bits, top[None]])
    q = rng.integers(0x3C00, 0x3F80, (B, 4, H, D)).astype(np.uint16)
    kb = rng.integers(0x3C00, 0x3F80, (B, 4, H, D)).astype(np.uint16)
    pl, bl = np.array([33, 7], np.int32), np.array([4, 2], np.int32)
    for kap, nu in [(1, 3), (2, 2), (3, 3), (1, 1)]:
        o1, l1 = oracle.attention_f8(top, top, codes, codes, 0, kap, nu, pl, bl, q, kb, kb)
        o2, l2 = oracle.attention(K, K, 0, kap, nu, pl, bl, q, kb, kb)
        assert np.array_equal(o1, o2) and np.array_equal(l1, l2)


def test_e4m3_append_rounds_low_depths_and_copies_the_top():
    rng = np.random.default_rng(23)
    R, L, B, cap, H, D, W = 3, 2, 2, 10, 1, 8, 4
    kt = rng.integers(0, 65535, (L, B, cap, H, D)).astype(np.uint16)
    kl = rng.integers(0, 255, (R - 1, L, B, cap, H, D)).astype(np.uint8)
    x = rng.normal(0, 3, (R, L, B, W, H, D)).astype(np.float32)
    kn = (x.view(np.uint32) >> 16).astype(np.uint16)
    acc, pl = np.array([1, 5], np.int32), np.array([2, 6], np.int32)
    kt2, vt2, kl2, vl2, pl2, flag = oracle.kv_append_f8(kt, kt, kl, kl, kn, kn, acc, pl)
    n = [2, 4]
    assert flag == 0 and list(pl2) == [4, 10]
    ekt, ekl = kt.copy(), kl.copy()
    for b in range(B):
        ekt[:, b, pl[b]:pl[b] + n[b]] = kn[R - 1, :, b, :n[b]]
        ekl[:, :, b, pl[b]:pl[b] + n[b]] = oracle.e4m3_from_bf16(kn[:R - 1, :, b, :n[b]])
    assert np.array_equal(kt2, ekt) and np.array_equal(kl2, ekl)
