"""Pins the oracle to facts that do not come from the oracle itself.

* Table 2 (Sec. 4.2): m*g head totals of the nine Pythia-160M variants, via the Eq. 18 block map.
* Table 1 (Sec. 3): OPT-175B cache-size ratios (exact) and the printed absolutes.
* Abstract / Sec. 6: MLKV-2 holds a 6x smaller cache than MQA-12.
* MHA (Sec. 2.1) and GQA / MQA (Secs. 2.2-2.3) against torch's scaled_dot_product_attention,
  a library routine, in float64.
* MLKV (Sec. 3) equals MHA run on explicitly duplicated K/V, bit for bit.
* Closed forms: one visible position, equal keys, zero query, one dominant key.
* Brute force on tiny inputs in 50-digit decimal arithmetic, without max subtraction.
* Prefill: torch's scaled_dot_product_attention with its causal mask, in float64, per prompt; the
  first prompt position returns its value row; MLKV prefill equals MHA prefill on duplicated K/V.
* KV-weight merge (Sec. 4.2): the identity map returns its input; a weight linear in (layer,
  head, element) merges to the closed form at the block's and group's mean layer and head;
  members permuted inside a block or group change nothing; blocks do not see each other.
* bfloat16 rounding: torch's float32 -> bfloat16 conversion (round to nearest even) on float32
  values, a brute-force nearest value over all 65,536 patterns on float64 values, and worked ties,
  subnormals and overflow.
"""
import decimal
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rows(fname):
    rows = []
    with open(os.path.join(GOLDEN, fname)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


# ----------------------------------------------------------------------------------------------
# maps and sizes
# ----------------------------------------------------------------------------------------------

def test_table2_total_kv_heads():
    rows = _rows("table2_pythia160m_variants.txt")
    assert len(rows) == 9
    for name, l, h, m, g, total in rows:
        l, h, m, g, total = map(int, (l, h, m, g, total))
        owner = oracle.block_owner_map(l, m)
        assert oracle.validate(owner, h, g) == 0, name
        m_found, slot = oracle.slots(owner)
        assert m_found == m, name
        assert m_found * g == total, name
        # the cache holds 2 * total heads per (sequence, position, channel)
        assert oracle.cache_elements(1, 1, m_found, g, 1) == 2 * total, name
        # every layer is mapped to a valid owner slot
        assert sorted(set(slot.tolist())) == list(range(m)), name


def test_table1_opt175b_ratios_and_printed_values():
    rows = {r[0]: (int(r[1]), int(r[2]), float(r[3])) for r in _rows("table1_opt175b.txt")}
    b, s, dk = 8, 1024, 128
    mha_m, mha_g, mha_gb = rows["MHA"]
    mha = oracle.cache_elements(b, s, mha_m, mha_g, dk)
    for method, (m, g, printed) in rows.items():
        e = oracle.cache_elements(b, s, m, g, dk)
        assert Fraction(e, mha) == Fraction(printed) / Fraction(mha_gb), method
        # printed absolutes: 8 bytes per element, GiB (the reading recorded with the fixture)
        assert Fraction(e * 8, 2 ** 30) == Fraction(printed), method
    # Sec. 2.5 formulas by name: MHA 2bslhd, GQA 2bslgd, MQA 2bsld
    assert mha == 2 * b * s * 96 * 96 * dk
    assert oracle.cache_elements(b, s, 96, 1, dk) * 96 == mha


def test_abstract_six_times_smaller_than_mqa():
    # MQA-12 (m=12, g=1) against MLKV-2 (m=2, g=1), Table 2 shapes
    mqa = oracle.cache_elements(64, 2048, 12, 1, 64)
    mlkv2 = oracle.cache_elements(64, 2048, 2, 1, 64)
    assert mqa == 6 * mlkv2


@pytest.mark.parametrize("l", [1, 2, 6, 12, 24, 32])
def test_block_map_structure(l):
    for m in range(1, l + 1):
        if l % m:
            with pytest.raises(ValueError):
                oracle.block_owner_map(l, m)
            continue
        owner = oracle.block_owner_map(l, m).tolist()
        per = l // m
        # contiguous blocks of l/m layers, each served by its bottom (first) layer
        assert owner == [n - n % per for n in range(l)]
        assert oracle.validate(owner, 4, 1) == 0
        assert oracle.slots(owner)[0] == m
    # m = l: every layer owns itself (MHA / GQA / MQA keep per-layer KV heads)
    assert oracle.block_owner_map(l, l).tolist() == list(range(l))
    # m = 1: one KV set for the whole model (MLKV-1)
    assert oracle.block_owner_map(l, 1).tolist() == [0] * l


@pytest.mark.parametrize("h", [1, 2, 3, 4, 6, 8, 12, 16, 32])
def test_group_map(h):
    for g in range(1, h + 1):
        if h % g:
            continue
        js = [oracle.kv_head_of(h, g, i) for i in range(h)]
        # each KV head serves h/g consecutive query heads
        assert js == sorted(js)
        assert [js.count(j) for j in range(g)] == [h // g] * g
    assert [oracle.kv_head_of(h, h, i) for i in range(h)] == list(range(h))   # MHA
    assert [oracle.kv_head_of(h, 1, i) for i in range(h)] == [0] * h          # MQA


def test_validate_rejects_bad_maps():
    assert oracle.validate([0, 0, 2, 2], 4, 2) == 0
    assert oracle.validate([0, 2, 2, 2], 4, 2) == oracle.ORACLE_ERR_MAP      # owner after layer
    assert oracle.validate([0, 0, 1, 1], 4, 2) == oracle.ORACLE_ERR_MAP      # owner not an owner
    assert oracle.validate([1, 1], 4, 2) == oracle.ORACLE_ERR_MAP            # owner[0] > 0
    assert oracle.validate([0, 0], 6, 4) == oracle.ORACLE_ERR_MAP            # g does not divide h
    assert oracle.validate([0, 0], 4, 8) == oracle.ORACLE_ERR_MAP            # g > h
    assert oracle.validate([0, 0], 4, 0) == oracle.ORACLE_ERR_ARG
    assert oracle.validate([-1, 0], 4, 1) == oracle.ORACLE_ERR_MAP


# ----------------------------------------------------------------------------------------------
# attention against torch's SDPA (library routine)
# ----------------------------------------------------------------------------------------------

def _random_problem(rng, owner, h, g, d, b, max_seq, seq_lens):
    c = oracle.OracleCache(owner, h, g, d, b, max_seq)
    for n in c.K:
        c.K[n][:] = rng.standard_normal(c.K[n].shape)
        c.V[n][:] = rng.standard_normal(c.V[n].shape)
    Q = {n: rng.standard_normal((b, h, d)) for n in range(len(owner))}
    return c, Q


def _sdpa_reference(c, layer, Q, seq_lens):
    """torch SDPA per sequence with the owner's KV heads repeated h/g times (float64)."""
    own = int(c.owner[layer])
    G = c.h // c.g
    out = np.zeros((c.b, c.h, c.d))
    for beta in range(c.b):
        L = int(seq_lens[beta])
        k = torch.from_numpy(c.K[own][beta, :, :L, :])           # [g][L][d]
        v = torch.from_numpy(c.V[own][beta, :, :L, :])
        k = torch.repeat_interleave(k, G, dim=0)                  # [h][L][d]
        v = torch.repeat_interleave(v, G, dim=0)
        q = torch.from_numpy(Q[beta]).unsqueeze(1)                # [h][1][d]
        o = torch.nn.functional.scaled_dot_product_attention(q[None], k[None], v[None])
        out[beta] = o[0, :, 0, :].numpy()
    return out


MAPS = [
    ("mha", [0, 1, 2], 4, 4),
    ("gqa", [0, 1, 2], 4, 2),
    ("mqa", [0, 1, 2], 4, 1),
    ("mlkv-block", [0, 0, 2, 2], 6, 3),
    ("mlkv-1", [0, 0, 0], 4, 1),
    ("non-uniform", [0, 0, 0, 3, 4, 4], 4, 2),
]


@pytest.mark.parametrize("name,owner,h,g", MAPS)
def test_oracle_matches_sdpa(name, owner, h, g):
    rng = np.random.default_rng(7)
    d, b, max_seq = 16, 3, 20
    seq_lens = np.array([1, 7, 20], dtype=np.int32)
    c, Q = _random_problem(rng, owner, h, g, d, b, max_seq, seq_lens)
    for layer in range(len(owner)):
        got = c.decode(layer, Q[layer], seq_lens)
        ref = _sdpa_reference(c, layer, Q[layer], seq_lens)
        np.testing.assert_allclose(got, ref, rtol=0, atol=1e-13)


def test_threads_do_not_change_results():
    rng = np.random.default_rng(3)
    owner, h, g, d, b, max_seq = [0, 0, 2], 6, 2, 8, 7, 33
    seq_lens = rng.integers(1, max_seq + 1, size=b).astype(np.int32)
    c, Q = _random_problem(rng, owner, h, g, d, b, max_seq, seq_lens)
    for layer in range(3):
        a = c.decode(layer, Q[layer], seq_lens, nthreads=1)
        z = c.decode(layer, Q[layer], seq_lens, nthreads=4)
        assert np.array_equal(a, z)


def test_mlkv_equals_mha_on_duplicated_kv():
    """Sec. 3: an MLKV layer computes what an MHA layer computes when every query head is given
    its own copy of the shared KV head (same layer's owner, same group)."""
    rng = np.random.default_rng(11)
    owner, h, g, d, b, max_seq = [0, 0, 0, 3, 3, 5], 6, 2, 8, 2, 9
    seq_lens = np.array([4, 9], dtype=np.int32)
    c, Q = _random_problem(rng, owner, h, g, d, b, max_seq, seq_lens)
    l = len(owner)
    mha = oracle.OracleCache(list(range(l)), h, h, d, b, max_seq)
    G = h // g
    for n in range(l):
        own = owner[n]
        for i in range(h):
            mha.K[n][:, i] = c.K[own][:, i // G]
            mha.V[n][:, i] = c.V[own][:, i // G]
    for n in range(l):
        assert np.array_equal(c.decode(n, Q[n], seq_lens), mha.decode(n, Q[n], seq_lens))


# ----------------------------------------------------------------------------------------------
# closed forms
# ----------------------------------------------------------------------------------------------

def test_single_position_returns_value_row():
    rng = np.random.default_rng(5)
    owner, h, g, d, b, max_seq = [0, 0], 4, 2, 8, 2, 5
    c, Q = _random_problem(rng, owner, h, g, d, b, max_seq, None)
    seq_lens = np.array([1, 1], dtype=np.int32)
    for n in range(2):
        out = c.decode(n, Q[n], seq_lens)
        for i in range(h):
            assert np.array_equal(out[:, i], c.V[0][:, i // 2, 0])


def test_equal_keys_and_zero_query_average_values():
    rng = np.random.default_rng(6)
    owner, h, g, d, b, max_seq = [0], 2, 1, 8, 1, 50
    c, Q = _random_problem(rng, owner, h, g, d, b, max_seq, None)
    c.K[0][:] = rng.standard_normal(d)                 # every position holds the same key
    seq_lens = np.array([37], dtype=np.int32)
    out = c.decode(0, Q[0], seq_lens)
    mean_v = c.V[0][0, 0, :37].mean(axis=0)
    np.testing.assert_allclose(out[0, 0], mean_v, rtol=0, atol=1e-15)
    np.testing.assert_allclose(out[0, 1], mean_v, rtol=0, atol=1e-15)
    # zero query: all scores 0, uniform weights whatever the keys
    c.K[0][:] = rng.standard_normal(c.K[0].shape)
    out0 = c.decode(0, np.zeros((1, h, d)), seq_lens)
    np.testing.assert_allclose(out0[0, 0], mean_v, rtol=0, atol=1e-15)


def test_dominant_key_selects_its_value():
    rng = np.random.default_rng(8)
    owner, h, g, d, b, max_seq = [0], 1, 1, 16, 1, 64
    c, Q = _random_problem(rng, owner, h, g, d, b, max_seq, None)
    q = np.zeros((1, 1, d))
    q[0, 0, 0] = 1.0
    c.K[0][0, 0, :, 0] = 0.0
    t_star = 41
    c.K[0][0, 0, t_star, 0] = 60.0 * np.sqrt(d)       # score gap 60 after the 1/sqrt(d) scale
    out = c.decode(0, q, np.array([64], dtype=np.int32))
    np.testing.assert_allclose(out[0, 0], c.V[0][0, 0, t_star], rtol=0, atol=1e-20)
    # the dominant key beyond the visible length is ignored
    out_short = c.decode(0, q, np.array([t_star], dtype=np.int32))
    np.testing.assert_allclose(out_short[0, 0], c.V[0][0, 0, :t_star].mean(axis=0), atol=1e-15)


# ----------------------------------------------------------------------------------------------
# brute force
# ----------------------------------------------------------------------------------------------

def test_brute_force_decimal():
    """Tiny MLKV problem: softmax written out with exp() of the raw scores (no max subtraction)
    and every operation in 50-digit decimal arithmetic."""
    decimal.getcontext().prec = 50
    D = decimal.Decimal
    rng = np.random.default_rng(13)
    owner, h, g, d, b, max_seq = [0, 0, 2], 4, 2, 3, 2, 5
    seq_lens = np.array([3, 5], dtype=np.int32)
    c, Q = _random_problem(rng, owner, h, g, d, b, max_seq, seq_lens)
    for n in range(3):
        got = c.decode(n, Q[n], seq_lens)
        Kown, Vown = c.K[owner[n]], c.V[owner[n]]
        for beta in range(b):
            for i in range(h):
                j = i // (h // g)
                scale = D(1) / D(d).sqrt()
                w = []
                for t in range(int(seq_lens[beta])):
                    s = sum(D(float(Q[n][beta, i, e])) * D(float(Kown[beta, j, t, e]))
                            for e in range(d))
                    w.append((s * scale).exp())
                Z = sum(w)
                for e in range(d):
                    ref = sum(wt * D(float(Vown[beta, j, t, e])) for t, wt in enumerate(w)) / Z
                    assert abs(float(ref) - got[beta, i, e]) < 1e-14


# ----------------------------------------------------------------------------------------------
# append
# ----------------------------------------------------------------------------------------------

def test_append_only_for_owner_layers():
    rng = np.random.default_rng(2)
    owner, h, g, d, b, max_seq = [0, 0, 2], 4, 2, 4, 2, 6
    c = oracle.OracleCache(owner, h, g, d, b, max_seq)
    seq_lens = np.array([3, 6], dtype=np.int32)
    K1, V1 = rng.standard_normal((b, g, d)), rng.standard_normal((b, g, d))
    before = {n: (c.K[n].copy(), c.V[n].copy()) for n in c.K}
    assert c.append(1, K1, V1, seq_lens) == 0                    # layer 1 owns nothing
    for n in c.K:
        assert np.array_equal(c.K[n], before[n][0]) and np.array_equal(c.V[n], before[n][1])
    assert c.append(2, K1, V1, seq_lens) == 1
    for beta in range(b):
        t = seq_lens[beta] - 1
        assert np.array_equal(c.K[2][beta, :, t], K1[beta])
        assert np.array_equal(c.V[2][beta, :, t], V1[beta])
        c.K[2][beta, :, t] = 0.0
        c.V[2][beta, :, t] = 0.0
    assert not c.K[2].any() and not c.V[2].any()               # nothing else was written
    assert not c.K[0].any()


# ----------------------------------------------------------------------------------------------
# prefill (causal attention over a whole prompt)
# ----------------------------------------------------------------------------------------------

def _prefill_problem(rng, owner, h, g, d, b, s_max, prompt_lens):
    c = oracle.OracleCache(owner, h, g, d, b, s_max)
    for n in sorted(set(owner)):
        c.load_prefix(n, rng.standard_normal((b, g, s_max, d)), rng.standard_normal((b, g, s_max, d)),
                      s_max)
    Q = rng.standard_normal((len(owner), b, s_max, h, d))
    return c, Q


@pytest.mark.parametrize("name,owner,h,g", MAPS)
def test_prefill_matches_causal_sdpa(name, owner, h, g):
    rng = np.random.default_rng(17)
    d, b, s_max = 16, 3, 23
    prompt_lens = np.array([1, 9, 23], dtype=np.int32)
    c, Q = _prefill_problem(rng, owner, h, g, d, b, s_max, prompt_lens)
    G = h // g
    for layer in range(len(owner)):
        got = c.prefill(layer, Q[layer], prompt_lens)
        own = owner[layer]
        for beta in range(b):
            S = int(prompt_lens[beta])
            k = torch.repeat_interleave(torch.from_numpy(c.K[own][beta, :, :S, :]), G, dim=0)
            v = torch.repeat_interleave(torch.from_numpy(c.V[own][beta, :, :S, :]), G, dim=0)
            q = torch.from_numpy(np.ascontiguousarray(Q[layer][beta, :S].transpose(1, 0, 2)))
            o = torch.nn.functional.scaled_dot_product_attention(q[None], k[None], v[None],
                                                                 is_causal=True)
            np.testing.assert_allclose(got[beta, :S], o[0].numpy().transpose(1, 0, 2), rtol=0,
                                       atol=1e-13)
            assert not got[beta, S:].any()


def test_prefill_first_position_returns_value_row():
    rng = np.random.default_rng(19)
    owner, h, g, d, b, s_max = [0, 0], 4, 2, 8, 2, 6
    c, Q = _prefill_problem(rng, owner, h, g, d, b, s_max, None)
    prompt_lens = np.array([6, 3], dtype=np.int32)
    for layer in range(2):
        got = c.prefill(layer, Q[layer], prompt_lens)
        for i in range(h):
            np.testing.assert_array_equal(got[:, 0, i], c.V[0][:, i // 2, 0])


def test_prefill_mlkv_equals_mha_on_duplicated_kv():
    rng = np.random.default_rng(23)
    owner, h, g, d, b, s_max = [0, 0, 2, 2], 6, 3, 8, 2, 11
    prompt_lens = np.array([11, 5], dtype=np.int32)
    c, Q = _prefill_problem(rng, owner, h, g, d, b, s_max, prompt_lens)
    mha = oracle.OracleCache(list(range(4)), h, h, d, b, s_max)
    G = h // g
    for n in range(4):
        for i in range(h):
            mha.K[n][:, i] = c.K[owner[n]][:, i // G]
            mha.V[n][:, i] = c.V[owner[n]][:, i // G]
    for n in range(4):
        assert np.array_equal(c.prefill(n, Q[n], prompt_lens), mha.prefill(n, Q[n], prompt_lens))


# ----------------------------------------------------------------------------------------------
# KV-weight merge (Sec. 4.2) and bfloat16 rounding
# ----------------------------------------------------------------------------------------------

def test_merge_identity_map_returns_input():
    # Every layer its own owner and g = h: every merged head has one member, itself.
    rng = np.random.default_rng(31)
    W = rng.standard_normal((5, 6, 40))
    np.testing.assert_array_equal(oracle.merge_kv(list(range(5)), 6, 6, W), W)


def _linear_weights(l, h, row):
    n = np.arange(l, dtype=np.float64)[:, None, None]
    i = np.arange(h, dtype=np.float64)[None, :, None]
    r = np.arange(row, dtype=np.float64)[None, None, :]
    return 1000.0 * n + 10.0 * i + 0.25 * r


@pytest.mark.parametrize("owner,h,g", [
    ([0, 0, 0, 3, 3, 3], 12, 4),          # Eq. 18 blocks of 3, GQA-4 inside
    ([0, 0, 2, 2, 4, 4, 6, 6], 8, 1),     # blocks of 2, one KV head
    ([0, 0, 0, 0, 4, 5, 5], 6, 3),        # blocks of 4, 1 and 2
])
def test_merge_linear_closed_form(owner, h, g):
    # W = 1000 n + 10 i + r/4 is linear, so its mean over a block B and a group J is
    # 1000 mean(B) + 10 mean(J) + r/4, with mean(J) = jG + (G-1)/2 for the contiguous group of Eq. 12.
    l, row, G = len(owner), 7, h // g
    out = oracle.merge_kv(owner, h, g, _linear_weights(l, h, row))
    owners = sorted(set(owner))
    for s_, o in enumerate(owners):
        block = [n for n in range(l) if owner[n] == o]
        for j in range(g):
            expect = 1000.0 * (sum(block) / len(block)) + 10.0 * (j * G + (G - 1) / 2) + \
                0.25 * np.arange(row)
            np.testing.assert_allclose(out[s_, j], expect, rtol=0, atol=1e-9)


def test_merge_permutation_invariance_and_locality():
    owner, h, g = [0, 0, 0, 3, 3], 8, 2
    rng = np.random.default_rng(32)
    W = rng.standard_normal((5, 8, 16))
    base = oracle.merge_kv(owner, h, g, W)
    P = W.copy()
    P[[0, 1, 2]] = W[[2, 0, 1]]                 # layers permuted inside block 0
    P[:, [4, 5, 6, 7]] = W[:, [7, 5, 4, 6]]     # heads permuted inside group 1
    np.testing.assert_allclose(oracle.merge_kv(owner, h, g, P), base, rtol=0, atol=1e-12)
    Q = W.copy()
    Q[3:] += 5.0                                # block 1 changes, block 0 does not see it
    out = oracle.merge_kv(owner, h, g, Q)
    np.testing.assert_array_equal(out[0], base[0])
    np.testing.assert_allclose(out[1], base[1] + 5.0, rtol=0, atol=1e-12)


def test_bf16_rne_matches_torch_on_float32_values():
    rng = np.random.default_rng(33)
    x = np.concatenate([
        rng.standard_normal(20000).astype(np.float32),
        (rng.standard_normal(5000) * 1e-39).astype(np.float32),      # float32 / bf16 subnormals
        (rng.standard_normal(5000) * 3e38).astype(np.float32),       # near overflow
        np.array([0.0, -0.0, 1.0, -1.0, 3.3895314e38, 3.4e38], dtype=np.float32),
    ])
    x = x[np.isfinite(x)]
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(oracle.bf16_rne(x.astype(np.float64)), ref)


def _all_bf16_values():
    bits = np.arange(65536, dtype=np.uint32)
    f = (bits << 16).astype(np.uint32).view(np.float32).astype(np.float64)
    ok = np.isfinite(f)
    return bits[ok].astype(np.uint16), f[ok]


def test_bf16_rne_brute_force_on_float64_values():
    bits, vals = _all_bf16_values()
    order = np.argsort(vals, kind="stable")
    bits, vals = bits[order], vals[order]
    rng = np.random.default_rng(34)
    x = np.concatenate([rng.standard_normal(300) * 10.0 ** rng.integers(-40, 38, 300),
                        rng.uniform(-3.0, 3.0, 300)])
    got = oracle.bf16_rne(x)
    for xv, gb in zip(x, got):
        d = np.abs(vals - xv)
        best = np.flatnonzero(d == d.min())
        cands = [int(bits[k]) for k in best if not (vals[k] == 0.0 and bits[k] == 0x8000)]
        if len(cands) > 1:     # a tie: the even significand
            cands = [c for c in cands if c % 2 == 0]
        if xv < 0 and vals[best[0]] == 0.0:
            cands = [0x8000]
        assert int(gb) == cands[0], (xv, hex(int(gb)), [hex(c) for c in cands])


def test_bf16_rne_worked_cases():
    cases = [
        (1.0, 0x3F80), (1.0 + 2.0 ** -8, 0x3F80),           # tie, even stays
        (1.0 + 3 * 2.0 ** -8, 0x3F82),                       # tie, rounds up to even
        (1.0 + 2.0 ** -8 + 2.0 ** -40, 0x3F81),              # just above the tie
        (-0.0, 0x8000), (0.0, 0x0000),
        (2.0 ** -133, 0x0001), (2.0 ** -134, 0x0000),        # smallest subnormal; tie to 0
        (3 * 2.0 ** -134, 0x0002), (-(2.0 ** -126), 0x8080),
        ((2 - 2.0 ** -7) * 2.0 ** 127, 0x7F7F),              # largest finite
        ((2 - 2.0 ** -8) * 2.0 ** 127, 0x7F80),              # tie at the top: overflows
        (1e300, 0x7F80), (-1e300, 0xFF80),
    ]
    for x, want in cases:
        assert int(oracle.bf16_rne(np.array([x]))[0]) == want, (x, want)
