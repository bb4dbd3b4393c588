"""Pins that tie the CPU oracle to something other than itself.

Each test checks the oracle against what the mathematics or the paper fixes:
dense softmax attention through numpy/scipy, closed forms, invariants, the
paper's printed sizes, and the published outputs of splitmix64. A plausible
mistake in the oracle (a dropped scale, a wrong kv-head mapping, a transposed
index, a wrong slot in a block) fails at least one of them.
"""
import math
import os

import numpy as np
import pytest
import scipy.special

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def f32(bits):
    return synth.bf16_bits_to_f32_np(bits).astype(np.float64)


def bf16(x):
    a = np.asarray(x, dtype=np.float32)
    return synth.f32_to_bf16_bits_np(a).reshape(a.shape)


def dense_attention(q_bits, k_bits, v_bits, scale, group):
    """Plain attention for one session/layer: q [Hq][D], k/v [Hkv][T][D]."""
    q, k, v = f32(q_bits), f32(k_bits), f32(v_bits)
    out = np.zeros_like(q)
    for h in range(q.shape[0]):
        g = h // group
        s = scale * (k[g] @ q[h])
        out[h] = scipy.special.softmax(s) @ v[g]
    return out


def make_case(seed, lens, L=2, Hq=8, Hkv=2, D=128, bt=16, spare=5, k_scale=1.0, poison=True):
    sess = list(range(len(lens)))
    nb = int(sum(-(-t // bt) for t in lens)) + spare
    tables = synth.random_block_tables(seed, lens, bt, nb)
    hot = synth.hot_pool_np(seed, sess, lens, tables, nb, L, Hkv, D, bt, k_scale, poison)
    q = synth.queries_np(seed, sess, range(L), Hq, D)
    return sess, tables, hot, q


@pytest.mark.parametrize("bt", [16, 4])
def test_paged_matches_dense_bruteforce(bt):
    lens = [37, 70, 16]
    L, Hq, Hkv, D = 2, 8, 2, 128
    scale = 1 / math.sqrt(D)
    sess, tables, hot, q = make_case(11, lens, L, Hq, Hkv, D, bt)
    out = oracle.paged_decode(hot, q, tables, lens, scale, Hq)
    for l in range(L):
        for b, T in enumerate(lens):
            k, v = synth.session_kv_np(11, sess[b], [l], Hkv, D, T)
            ref = dense_attention(q[l, b], k[0], v[0], scale, Hq // Hkv)
            np.testing.assert_allclose(out[l, b], ref, rtol=1e-10, atol=1e-12)


def test_paged_matches_dense_on_drawn_shapes():
    """The same brute-force pin over drawn shapes: group sizes from MHA to
    8 q-heads per kv-head, block sizes 1 to 32, head dims 16 to 128, ragged
    lengths from one token up, and scales including the config-1 reading."""
    hyp = pytest.importorskip("hypothesis")
    st = hyp.strategies

    @hyp.settings(max_examples=30, deadline=None, derandomize=True)
    @hyp.given(hk=st.sampled_from([(4, 4), (8, 2), (8, 1), (6, 3), (32, 4)]),
               bt=st.sampled_from([1, 4, 16, 32]), D=st.sampled_from([16, 64, 128]),
               lens=st.lists(st.integers(1, 80), min_size=1, max_size=3),
               scale=st.sampled_from([1.0, 1 / math.sqrt(128), 0.3]),
               seed=st.integers(0, 1000))
    def check(hk, bt, D, lens, scale, seed):
        Hq, Hkv = hk
        sess, tables, hot, q = make_case(seed, lens, 1, Hq, Hkv, D, bt)
        out = oracle.paged_decode(hot, q, tables, lens, scale, Hq)
        for b, T in enumerate(lens):
            k, v = synth.session_kv_np(seed, sess[b], [0], Hkv, D, T)
            ref = dense_attention(q[0, b], k[0], v[0], scale, Hq // Hkv)
            np.testing.assert_allclose(out[0, b], ref, rtol=1e-10, atol=1e-12)

    check()


def test_layer_offset_selects_layer():
    lens = [40, 9]
    sess, tables, hot, q = make_case(3, lens, L=3)
    full = oracle.paged_decode(hot, q, tables, lens, 0.1, 8)
    one = oracle.paged_decode(hot, q[2:3], tables, lens, 0.1, 8, layer0=2)
    assert np.array_equal(full[2:3], one)


def test_one_token_returns_value_row():
    lens = [1, 1]
    L, Hq, Hkv, D = 1, 8, 2, 128
    sess, tables, hot, q = make_case(5, lens, L, Hq, Hkv, D)
    out = oracle.paged_decode(hot, q, tables, lens, 0.7, Hq)
    for b in range(2):
        _, v = synth.session_kv_np(5, sess[b], [0], Hkv, D, 1)
        for h in range(Hq):
            assert np.array_equal(out[0, b, h], f32(v[0, h // 4, 0]))


def test_equal_keys_give_mean_of_values():
    T, L, Hq, Hkv, D, bt = 45, 1, 8, 2, 128, 16
    sess, tables, hot, q = make_case(9, [T], L, Hq, Hkv, D, bt)
    key_row = bf16(np.linspace(-1, 1, D))
    for j in range(-(-T // bt)):
        hot[tables[0, j], :, 0, :, :, :] = key_row
    out = oracle.paged_decode(hot, q, tables, [T], 0.3, Hq)
    _, v = synth.session_kv_np(9, 0, [0], Hkv, D, T)
    for h in range(Hq):
        np.testing.assert_allclose(out[0, 0, h], f32(v[0, h // 4]).mean(axis=0), rtol=0, atol=1e-12)


def test_two_token_logistic_closed_form():
    # q = e_0, k_0 = a e_0, k_1 = b e_0: weights are the logistic of scale*(a-b).
    D, bt = 128, 16
    a, b, scale = 1.5, -0.25, 0.8
    hot = np.zeros((2, 1, 2, 1, bt, D), dtype=np.uint16)
    hot[1, 0, 0, 0, 0, 0] = bf16(a)
    hot[1, 0, 0, 0, 1, 0] = bf16(b)
    v0 = bf16(np.arange(D) / 64.0 - 1.0)
    v1 = bf16(np.cos(np.arange(D)))
    hot[1, 0, 1, 0, 0] = v0
    hot[1, 0, 1, 0, 1] = v1
    q = np.zeros((1, 1, 1, D), dtype=np.uint16)
    q[0, 0, 0, 0] = bf16(1.0)
    out = oracle.paged_decode(hot, q, np.array([[1]], dtype=np.int32), [2], scale, 1)
    w0 = 1.0 / (1.0 + math.exp(-scale * (a - b)))
    ref = w0 * f32(v0) + (1 - w0) * f32(v1)
    np.testing.assert_allclose(out[0, 0, 0], ref, rtol=0, atol=1e-15)


def test_physical_permutation_is_bit_invariant():
    lens = [33, 64, 17, 5]
    sess, tables, hot, q = make_case(21, lens, spare=9)
    out1 = oracle.paged_decode(hot, q, tables, lens, 0.125, 8)
    rng = np.random.default_rng(4)
    perm = rng.permutation(hot.shape[0]).astype(np.int32)
    hot2 = np.empty_like(hot)
    hot2[perm] = hot
    t2 = np.where(tables >= 0, perm[np.maximum(tables, 0)], -1).astype(np.int32)
    out2 = oracle.paged_decode(hot2, q, t2, lens, 0.125, 8)
    assert np.array_equal(out1, out2)


def test_mha_special_case():
    lens = [29, 50]
    L, H, D = 1, 4, 128
    sess, tables, hot, q = make_case(2, lens, L, H, H, D)
    out = oracle.paged_decode(hot, q, tables, lens, 0.2, H)
    for b, T in enumerate(lens):
        k, v = synth.session_kv_np(2, b, [0], H, D, T)
        np.testing.assert_allclose(out[0, b], dense_attention(q[0, b], k[0], v[0], 0.2, 1),
                                   rtol=1e-10, atol=1e-12)


def test_nan_poisoned_tail_slots_are_ignored():
    lens = [19, 47]
    _, tables, hot_nan, q = make_case(8, lens, poison=True)
    _, _, hot_zero, _ = make_case(8, lens, poison=False)
    a = oracle.paged_decode(hot_nan, q, tables, lens, 0.125, 8)
    b = oracle.paged_decode(hot_zero, q, tables, lens, 0.125, 8)
    assert np.all(np.isfinite(a))
    assert np.array_equal(a, b)


def test_bad_arguments_rejected():
    lens = [20]
    _, tables, hot, q = make_case(1, lens, L=1)
    with pytest.raises(ValueError):
        oracle.paged_decode(hot, q, tables, [0], 0.1, 8)
    bad = tables.copy()
    bad[0, 0] = hot.shape[0]
    with pytest.raises(ValueError):
        oracle.paged_decode(hot, q, bad, lens, 0.1, 8)


# ---------------------------------------------------------------- migration

def image_as_blocks(img, T, bt):
    """numpy restatement: image rows grouped into bt-token blocks."""
    L, two, Hkv, cap, D = img.shape
    nb = -(-T // bt)
    pad = np.zeros((L, 2, Hkv, nb * bt, D), dtype=img.dtype)
    pad[:, :, :, :T] = img[:, :, :, :T]
    return pad.reshape(L, 2, Hkv, nb, bt, D).transpose(3, 0, 1, 2, 4, 5)


@pytest.mark.parametrize("T,bt", [(1, 16), (16, 16), (37, 16), (130, 64), (64, 64)])
def test_unpack_matches_reshape(T, bt):
    L, Hkv, D, cap = 3, 2, 128, 160
    img = synth.session_image_np(4, 7, L, Hkv, D, T, cap)
    nb = -(-T // bt)
    NB = nb + 6
    row = synth.random_block_tables(T, [T], bt, NB)[0]
    hot = np.zeros((NB, L, 2, Hkv, bt, D), dtype=np.uint16)
    oracle.unpack(img, T, row, hot)
    blocks = image_as_blocks(img, T, bt)
    for j in range(nb):
        n = min(bt, T - j * bt)
        assert np.array_equal(hot[row[j], :, :, :, :n], blocks[j][:, :, :, :n])
        assert not np.any(hot[row[j], :, :, :, n:])  # slots past T untouched
    untouched = np.setdiff1d(np.arange(NB), row[:nb])
    assert not np.any(hot[untouched])


def test_pack_unpack_round_trip_and_write_once():
    L, Hkv, D, bt, cap, T = 2, 4, 128, 16, 100, 83
    img = synth.session_image_np(6, 1, L, Hkv, D, T, cap, poison_tail=False)
    NB = 12
    row = synth.random_block_tables(2, [T], bt, NB)[0]
    hot = np.zeros((NB, L, 2, Hkv, bt, D), dtype=np.uint16)
    oracle.unpack(img, T, row, hot)
    img2 = np.zeros_like(img)
    written = oracle.pack(hot, row, 0, T, img2)
    assert np.array_equal(img2, img)
    assert written == T * oracle.kv_bytes_per_token(L, Hkv, D)
    # write-on-evict: tokens already in the image are not written again
    assert oracle.pack(hot, row, T, T, img2) == 0
    img3 = np.full_like(img, 7)
    written = oracle.pack(hot, row, 50, T, img3)
    assert written == (T - 50) * oracle.kv_bytes_per_token(L, Hkv, D)
    assert np.all(img3[:, :, :, :50] == 7)
    assert np.array_equal(img3[:, :, :, 50:T], img[:, :, :, 50:T])
    # unpack of the packed image restores the valid hot bytes
    hot2 = np.zeros_like(hot)
    oracle.unpack(img2, T, row, hot2)
    assert np.array_equal(hot2, hot)


def test_migration_copies_on_drawn_shapes():
    """Unpack against the image reshaped into blocks, pack(unpack(image)) ==
    image, and a pack from t0 writing exactly tokens [t0, T), over drawn
    layer counts, kv-head counts, block sizes, lengths and placements."""
    hyp = pytest.importorskip("hypothesis")
    st = hyp.strategies

    @hyp.settings(max_examples=30, deadline=None, derandomize=True)
    @hyp.given(L=st.integers(1, 3), Hkv=st.sampled_from([1, 2, 4]),
               bt=st.sampled_from([1, 4, 16, 64]), T=st.integers(1, 150),
               extra=st.integers(0, 40), t0_frac=st.floats(0.0, 1.0),
               seed=st.integers(0, 1000))
    def check(L, Hkv, bt, T, extra, t0_frac, seed):
        D, cap = 16, T + extra
        img = synth.session_image_np(seed, 3, L, Hkv, D, T, cap, poison_tail=False)
        nb = -(-T // bt)
        NB = nb + 3
        row = synth.random_block_tables(seed, [T], bt, NB)[0]
        hot = np.zeros((NB, L, 2, Hkv, bt, D), dtype=np.uint16)
        oracle.unpack(img, T, row, hot)
        blocks = image_as_blocks(img, T, bt)
        for j in range(nb):
            n = min(bt, T - j * bt)
            assert np.array_equal(hot[row[j], :, :, :, :n], blocks[j][:, :, :, :n])
        back = np.zeros_like(img)
        per_tok = oracle.kv_bytes_per_token(L, Hkv, D)
        assert oracle.pack(hot, row, 0, T, back) == T * per_tok
        assert np.array_equal(back[:, :, :, :T], img[:, :, :, :T])
        t0 = int(t0_frac * T)
        part = np.full_like(img, 0x5A5A)
        assert oracle.pack(hot, row, t0, T, part) == (T - t0) * per_tok
        assert np.all(part[:, :, :, :t0] == 0x5A5A) and np.all(part[:, :, :, T:] == 0x5A5A)
        assert np.array_equal(part[:, :, :, t0:T], img[:, :, :, t0:T])

    check()


def test_append_positions():
    L, Hkv, D, bt = 2, 2, 128, 16
    NB = 6
    row = np.array([4, 1, 3], dtype=np.int32)
    hot = np.zeros((NB, L, 2, Hkv, bt, D), dtype=np.uint16)
    pos0, n = 14, 20
    k, v = synth.session_kv_np(1, 3, range(L), Hkv, D, pos0 + n)
    kk = np.ascontiguousarray(k[:, :, pos0:, :].transpose(0, 2, 1, 3))   # [L][n][Hkv][D]
    vv = np.ascontiguousarray(v[:, :, pos0:, :].transpose(0, 2, 1, 3))
    oracle.append(hot, row, pos0, kk, vv)
    for t in range(pos0, pos0 + n):
        p, s = row[t // bt], t % bt
        assert np.array_equal(hot[p, :, 0, :, s], k[:, :, t])
        assert np.array_equal(hot[p, :, 1, :, s], v[:, :, t])
    assert not np.any(hot[row[0], :, :, :, :pos0])


# ------------------------------------------------------------------- sizes

def read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


def test_paper_sizes():
    g = {r[0]: float(r[1]) for r in read_golden("paper_sizes.txt")}
    per_tok = oracle.kv_bytes_per_token(48, 4, 128)
    assert per_tok == g["kv_bytes_per_token"] * 1024
    assert 16 * per_tok == g["block_bytes_16_tokens"] * 1024 ** 2
    peak = g["peak_context_tokens"] * 1000 * per_tok / 1024 ** 3
    assert abs(peak - g["peak_context_bytes"]) < 0.005


# -------------------------------------------------------------- placement

def test_splitmix64_published_outputs():
    for row in read_golden("splitmix64.txt"):
        seed, outs = int(row[0]), [int(x) for x in row[1:]]
        assert oracle.splitmix64_stream(seed, len(outs)) == outs


def test_fisher_yates_definition_small():
    # n = 2: one draw r; the swap happens iff floor(2 r / 2^64) == 0.
    for seed in range(40):
        r = oracle.splitmix64_stream(seed, 1)[0]
        got = oracle.shuffle(np.array([0, 1]), seed)
        j = (r * 2) >> 64
        assert list(got) == ([1, 0] if j == 0 else [0, 1])


def test_fisher_yates_uniform_on_four():
    counts = {}
    n_seeds = 24000
    for seed in range(n_seeds):
        p = tuple(oracle.shuffle(np.arange(4), seed * 7919 + 1))
        counts[p] = counts.get(p, 0) + 1
    assert len(counts) == 24
    exp = n_seeds / 24
    chi2 = sum((c - exp) ** 2 / exp for c in counts.values())
    assert chi2 < 60  # 23 dof; p < 1e-4 above ~55


def test_free_list_pop_push_contract():
    fl = oracle.FreeList(10, 99)
    start = fl.contents()
    assert sorted(start) == list(range(10))
    got = fl.pop(3)
    assert list(got) == list(start[::-1][:3])
    fl.push(got)
    assert list(fl.contents()) == list(start[:7]) + list(got)
    with pytest.raises(MemoryError):
        fl.pop(11)


def test_session_lengths_stay_in_range():
    """Lengths are draws on [lo, hi]; one is made ragged (not a multiple of
    the block size) only when [lo, hi] holds such a length."""
    for seed, n, lo, hi in [(0, 1, 65536, 65536), (1, 3, 16, 16), (2, 32, 8192, 32768),
                            (3, 4, 64, 65), (4, 8, 1, 2048), (5, 2, 32, 47)]:
        t = synth.session_lengths(seed, n, lo, hi, 16)
        assert len(t) == n and t.min() >= lo and t.max() <= hi
        if any(x % 16 for x in range(lo, hi + 1)):
            assert any(int(x) % 16 for x in t)
