"""Pins of the oracle's decode attention.

Anchors: single-token and equal-key closed forms, a two-token example computed by
hand, page-shuffle invariance, the grouped-query head mapping, torch's CPU
scaled_dot_product_attention in fp64, and the log-sum-exp split identity (the
shared-prefix merge equals attention over the concatenated KV).
"""
import numpy as np
import pytest

from oracle import attention
from oracle.sampling import bf16_bits_to_f32
from paper_2607_20791_gb300 import workloads
from paper_2607_20791_gb300.workloads import f32_to_bf16_bits


def _case(G=2, rpg=3, Hq=4, Hkv=2, D=16, plens=(20, 33), slens=(0, 5, 17, 1, 16, 40), seed=0):
    return workloads.make_attn_case("t", G, rpg, Hq, Hkv, D, plens, slens, seed)


def _tokens(case, r, h):
    g = r // case.rows_per_group
    kp = attention.gather_tokens(case.k_pages, case.prompt_block_table[g], int(case.prompt_len[g]), h, 16)
    ks = attention.gather_tokens(case.k_pages, case.suffix_block_table[r], int(case.suffix_len[r]), h, 16)
    vp = attention.gather_tokens(case.v_pages, case.prompt_block_table[g], int(case.prompt_len[g]), h, 16)
    vs = attention.gather_tokens(case.v_pages, case.suffix_block_table[r], int(case.suffix_len[r]), h, 16)
    return np.concatenate([kp, ks]), np.concatenate([vp, vs])


def test_single_token_returns_its_value():
    case = _case(G=1, rpg=1, plens=(1,), slens=(0,))
    o, lse = attention.decode_attention_case(case)
    for j in range(case.num_q_heads):
        h = j // 2
        K, V = _tokens(case, 0, h)
        assert np.array_equal(o[0, j], V[0])
        q = bf16_bits_to_f32(case.q[0, j]).astype(np.float64)
        assert lse[0, j] == pytest.approx(case.softmax_scale * float(K[0] @ q), abs=1e-12)


def test_equal_keys_average_values():
    case = _case(G=1, rpg=2, plens=(37,), slens=(3, 0))
    case.k_pages[:] = case.k_pages[0, 0, 0]  # every key identical
    o, lse = attention.decode_attention_case(case)
    for r in range(2):
        for j in range(case.num_q_heads):
            _, V = _tokens(case, r, j // 2)
            assert np.allclose(o[r, j], V.mean(axis=0), atol=1e-12)


def test_two_token_hand_example():
    # D = 2, scale = 1: q = (1, 0); k0 = (0, 0), k1 = (ln 3, 0) -> weights 1/4, 3/4
    D = 2
    case = workloads.make_attn_case("h", 1, 1, 1, 1, D, [2], [0], seed=0)
    case.softmax_scale = 1.0
    case.q[0, 0] = f32_to_bf16_bits(np.array([1.0, 0.0], np.float32))
    k = np.zeros((2, D), np.float32)
    lnq = float(bf16_bits_to_f32(f32_to_bf16_bits(np.array([np.log(3.0)], np.float32)))[0])
    k[1, 0] = lnq
    v = np.array([[4.0, -8.0], [8.0, 4.0]], np.float32)
    page = int(case.prompt_block_table[0, 0])
    case.k_pages[page, 0, :2] = f32_to_bf16_bits(k)
    case.v_pages[page, 0, :2] = f32_to_bf16_bits(v)
    o, lse = attention.decode_attention_case(case)
    w1 = np.exp(lnq) / (1.0 + np.exp(lnq))
    assert np.allclose(o[0, 0], (1 - w1) * v[0] + w1 * v[1], atol=1e-12)
    assert lse[0, 0] == pytest.approx(np.log(1.0 + np.exp(lnq)), abs=1e-12)
    assert w1 == pytest.approx(0.75, abs=2e-3)


def test_empty_kv_gives_zero_and_minus_inf():
    case = _case(G=1, rpg=2, plens=(0,), slens=(0, 4))
    o, lse = attention.decode_attention_case(case)
    assert np.all(o[0] == 0) and np.all(np.isneginf(lse[0]))
    assert np.all(np.isfinite(lse[1]))


def test_page_shuffle_invariance():
    case = _case()
    o1, l1 = attention.decode_attention_case(case)
    rng = np.random.default_rng(5)
    perm = rng.permutation(case.num_pages)  # new slot of old page p is perm[p]
    k2 = np.empty_like(case.k_pages)
    v2 = np.empty_like(case.v_pages)
    k2[perm] = case.k_pages
    v2[perm] = case.v_pages
    remap = lambda t: np.where(t >= 0, perm[np.maximum(t, 0)], -1).astype(np.int32)
    o2, l2 = attention.decode_attention(case.q, k2, v2, remap(case.prompt_block_table),
                                        case.prompt_len, remap(case.suffix_block_table),
                                        case.suffix_len, case.rows_per_group, case.num_kv_heads)
    assert np.array_equal(o1, o2) and np.array_equal(l1, l2)


def test_gqa_head_mapping():
    case = _case(Hq=6, Hkv=3)
    case.v_pages[:, [0, 2]] = 0  # only kv head 1 carries values
    o, _ = attention.decode_attention_case(case)
    assert np.all(o[:, [0, 1, 4, 5]] == 0)
    assert np.all(np.abs(o[:, [2, 3]]).sum(axis=-1) > 0)


def test_matches_torch_sdpa_fp64():
    torch = pytest.importorskip("torch")
    case = _case(G=3, rpg=2, Hq=8, Hkv=2, D=32, plens=(50, 0, 129), slens=(0, 7, 16, 33, 2, 64))
    o, lse = attention.decode_attention_case(case)
    q = bf16_bits_to_f32(case.q).astype(np.float64)
    for r in range(case.num_rows):
        for h in range(case.num_kv_heads):
            K, V = _tokens(case, r, h)
            if K.shape[0] == 0:
                continue
            qs = torch.from_numpy(q[r, h * 4:(h + 1) * 4])[None, :, None, :]   # [1, 4, 1, D]
            Kt = torch.from_numpy(K)[None, None].expand(1, 4, -1, -1)
            Vt = torch.from_numpy(V)[None, None].expand(1, 4, -1, -1)
            ref = torch.nn.functional.scaled_dot_product_attention(qs, Kt, Vt, scale=case.softmax_scale)
            assert np.allclose(o[r, h * 4:(h + 1) * 4], ref[0, :, 0].numpy(), atol=1e-12)
            s = case.softmax_scale * (torch.from_numpy(K) @ qs[0, :, 0].T)  # [T, 4]
            assert np.allclose(lse[r, h * 4:(h + 1) * 4], torch.logsumexp(s, dim=0).numpy(), atol=1e-12)


def test_paged_layout_against_dense_tokens():
    # the tokens are drawn first as dense [T, D] arrays in sequence order and then
    # scattered into the page pool by this test (token t of a sequence -> page
    # table[t // 16], slot t % 16); the oracle's gather must give attention over
    # the dense arrays (torch fp64), across page boundaries and partial last pages
    torch = pytest.importorskip("torch")
    G, rpg, Hq, Hkv, D = 2, 2, 4, 2, 16
    plens, slens = (37, 16), (0, 21, 5, 33)
    case = workloads.make_attn_case("dense", G, rpg, Hq, Hkv, D, plens, slens, seed=11)
    rng = np.random.default_rng(12)
    bf = lambda shape: f32_to_bf16_bits(rng.standard_normal(shape).astype(np.float32))
    case.k_pages[:] = 0
    case.v_pages[:] = 0
    dense = {}
    for kind, table, lens in (("p", case.prompt_block_table, plens), ("s", case.suffix_block_table, slens)):
        for i, n in enumerate(lens):
            K, V = bf((Hkv, n, D)), bf((Hkv, n, D))
            dense[kind, i] = (K, V)
            for t in range(n):
                case.k_pages[table[i, t // 16], :, t % 16] = K[:, t]
                case.v_pages[table[i, t // 16], :, t % 16] = V[:, t]
    o, lse = attention.decode_attention_case(case)
    q = bf16_bits_to_f32(case.q).astype(np.float64)
    for r in range(G * rpg):
        Kp, Vp = dense["p", r // rpg]
        Ks, Vs = dense["s", r]
        for j in range(Hq):
            h = j // (Hq // Hkv)
            K = bf16_bits_to_f32(np.concatenate([Kp[h], Ks[h]])).astype(np.float64)
            V = bf16_bits_to_f32(np.concatenate([Vp[h], Vs[h]])).astype(np.float64)
            qs = torch.from_numpy(q[r, j])[None, None, None, :]
            ref = torch.nn.functional.scaled_dot_product_attention(
                qs, torch.from_numpy(K)[None, None], torch.from_numpy(V)[None, None], scale=case.softmax_scale)
            assert np.allclose(o[r, j], ref[0, 0, 0].numpy(), atol=1e-12), (r, j)
            s = case.softmax_scale * (K @ q[r, j])
            assert lse[r, j] == pytest.approx(float(torch.logsumexp(torch.from_numpy(s), 0)), abs=1e-12)


def test_split_merge_identity():
    # attention over [prompt | suffix] = log-sum-exp merge of attention over each part
    case = _case(G=1, rpg=3, plens=(45,), slens=(9, 0, 31))
    o, lse = attention.decode_attention_case(case)
    empty_bt = np.full_like(case.suffix_block_table, -1)
    zeros = np.zeros_like(case.suffix_len)
    o_p, l_p = attention.decode_attention(case.q, case.k_pages, case.v_pages, case.prompt_block_table,
                                          case.prompt_len, empty_bt, zeros, 3, case.num_kv_heads)
    no_prompt = np.zeros_like(case.prompt_len)
    o_s, l_s = attention.decode_attention(case.q, case.k_pages, case.v_pages, case.prompt_block_table,
                                          no_prompt, case.suffix_block_table, case.suffix_len, 3,
                                          case.num_kv_heads)
    m = np.maximum(l_p, l_s)
    a = np.exp(l_p - m)
    b = np.where(np.isneginf(l_s), 0.0, np.exp(l_s - m))
    merged = (a[..., None] * o_p + b[..., None] * o_s) / (a + b)[..., None]
    assert np.allclose(merged, o, atol=1e-12)
    assert np.allclose(m + np.log(a + b), lse, atol=1e-12)
