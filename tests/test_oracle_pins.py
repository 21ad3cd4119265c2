"""Pins for the CPU oracle against things other than itself: library routines
(torch CPU fp64, scipy, numpy complex exponentials), closed forms, invariants
and the paper's printed numbers.  Each test is chosen so that a plausible slip
in the oracle (dropped term, wrong sign or index, transposed operand, wrong
pairing) fails it."""
import math

import numpy as np
import pytest
import scipy.special
import torch
import torch.nn.functional as F

import oracle
from conftest import read_golden
from paper_2606_13361_gb300 import inputs


# ------------------------------------------------------------------ bf16 ----

def _torch_bf16_bits(x32: np.ndarray) -> np.ndarray:
    t = torch.from_numpy(np.ascontiguousarray(x32, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def test_bf16_encode_matches_torch_on_fp32_values():
    rng = np.random.default_rng(1)
    with np.errstate(invalid="ignore", over="ignore"):
        x = _bf16_cases(rng)
    x = x[np.isfinite(x)]
    got = oracle.bf16_encode(x.astype(np.float64))
    want = _torch_bf16_bits(x)
    assert np.array_equal(got, want)


def _bf16_cases(rng):
    return np.concatenate([
        rng.standard_normal(20000).astype(np.float32) * 10.0 ** rng.integers(-30, 30, 20000),
        # exact ties: low 16 bits == 0x8000, both parities of the kept bit
        (rng.integers(0, 1 << 15, 4000).astype(np.uint32) << 17 | 0x8000
         | (rng.integers(0, 2, 4000).astype(np.uint32) << 16)).view(np.float32),
        # fp32 subnormals and the overflow edge
        (rng.integers(1, 1 << 23, 2000).astype(np.uint32)).view(np.float32),
        np.array([3.3895313892515355e38, 3.3961e38, -3.40e38, 0.0, -0.0], dtype=np.float32),
    ]).astype(np.float32)


def test_bf16_decode_is_exact_for_all_finite_patterns():
    h = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    vals = torch.from_numpy(h.view(np.int16)).view(torch.bfloat16).to(torch.float64).numpy()
    got = oracle.bf16_decode(h)
    fin = np.isfinite(vals)
    assert np.array_equal(got[fin], vals[fin])
    assert np.all(np.isinf(got[np.isinf(vals)]))


def test_bf16_roundtrip_of_decoded_values_is_identity():
    h = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    v = oracle.bf16_decode(h)
    fin = np.isfinite(v)
    back = oracle.bf16_encode(v[fin])
    # -0 and +0 keep their sign; every finite pattern maps to itself
    assert np.array_equal(back, h[fin])


# --------------------------------------------------------------- RMSNorm ----

@pytest.mark.parametrize("d", [64, 128])
def test_rmsnorm_matches_torch(d):
    rng = np.random.default_rng(2)
    x = rng.standard_normal((37, d)) * 3.0
    w = 1.0 + 0.1 * rng.standard_normal(d)
    eps = 1e-6
    got = oracle.rmsnorm(x, w, eps)
    want = F.rms_norm(torch.from_numpy(x), (d,), weight=torch.from_numpy(w), eps=eps).numpy()
    np.testing.assert_allclose(got, want, rtol=1e-13, atol=1e-14)
    # unit weight: output rms is 1 up to eps
    y1 = oracle.rmsnorm(x, np.ones(d), 0.0)
    np.testing.assert_allclose(np.sqrt(np.mean(y1 ** 2, axis=-1)), 1.0, rtol=1e-13)


# ------------------------------------------------------------------ RoPE ----

def _rope_complex(x, pos, theta):
    d = x.shape[-1]
    h = d // 2
    i = np.arange(h)
    ang = np.asarray(pos, dtype=np.float64)[..., None] * theta ** (-2.0 * i / d)
    z = (x[..., :h] + 1j * x[..., h:]) * np.exp(1j * ang)
    return np.concatenate([z.real, z.imag], axis=-1)


@pytest.mark.parametrize("d", [2, 64, 128])
def test_rope_matches_complex_rotation(d):
    rng = np.random.default_rng(3)
    x = rng.standard_normal((50, d))
    pos = rng.integers(0, 40000, 50)
    got = oracle.rope(x, pos, 1e6)
    np.testing.assert_allclose(got, _rope_complex(x, pos, 1e6), rtol=1e-11, atol=1e-11)


def test_rope_d2_closed_form_and_identity_at_zero():
    x = np.array([[0.3, -1.7]])
    for p in (0, 1, 5, 1000):
        got = oracle.rope(x, [p], 1e6)[0]
        want = [0.3 * math.cos(p) + 1.7 * math.sin(p), -1.7 * math.cos(p) + 0.3 * math.sin(p)]
        np.testing.assert_allclose(got, want, rtol=1e-13, atol=1e-15)
    y = np.random.default_rng(4).standard_normal((3, 128))
    assert np.array_equal(oracle.rope(y, [0, 0, 0], 1e6), y)


def test_rope_relative_position_invariance_and_norm():
    rng = np.random.default_rng(5)
    d = 128
    q, k = rng.standard_normal(d), rng.standard_normal(d)
    for (m, n, s) in [(10, 3, 100), (3774, 100, 28000), (0, 64, 7)]:
        a = oracle.rope(q[None], [m], 1e6)[0] @ oracle.rope(k[None], [n], 1e6)[0]
        b = oracle.rope(q[None], [m + s], 1e6)[0] @ oracle.rope(k[None], [n + s], 1e6)[0]
        assert abs(a - b) < 1e-9 * (1 + abs(a))
    r = oracle.rope(q[None], [31337], 1e6)[0]
    assert abs(np.linalg.norm(r) - np.linalg.norm(q)) < 1e-12


def test_rope_pairs_first_and_second_half():
    # rotate-half: only (i, i+d/2) mix; an input on one coordinate spills only
    # into its partner
    d = 16
    x = np.zeros((1, d))
    x[0, 3] = 1.0
    y = oracle.rope(x, [7], 1e6)[0]
    nz = set(np.flatnonzero(np.abs(y) > 0))
    assert nz <= {3, 3 + d // 2}
    ang = 7 * 1e6 ** (-2 * 3 / d)
    np.testing.assert_allclose([y[3], y[3 + d // 2]], [math.cos(ang), math.sin(ang)], rtol=1e-13)


# ------------------------------------------------------------- attention ----

def _sdpa(q, row_pos, k, v):
    """torch SDPA (fp64, CPU) with an explicit causal mask for the given row positions."""
    R, Hq, d = q.shape
    N, Hkv, _ = k.shape
    mask = torch.from_numpy(np.arange(N)[None, :] <= np.asarray(row_pos)[:, None])
    qt = torch.from_numpy(q).permute(1, 0, 2)[None]
    kt = torch.from_numpy(k).permute(1, 0, 2)[None]
    vt = torch.from_numpy(v).permute(1, 0, 2)[None]
    o = F.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask, enable_gqa=(Hq != Hkv))
    return o[0].permute(1, 0, 2).numpy()


@pytest.mark.parametrize("Hq,Hkv,d,N", [(4, 1, 64, 40), (8, 2, 32, 33), (3, 3, 16, 17), (32, 8, 128, 20)])
def test_attention_matches_torch_sdpa(Hq, Hkv, d, N):
    rng = np.random.default_rng(6)
    q = rng.standard_normal((N, Hq, d))
    k = rng.standard_normal((N, Hkv, d))
    v = rng.standard_normal((N, Hkv, d))
    pos = np.arange(N)
    o, lse = oracle.attention(q, pos, k, v)
    np.testing.assert_allclose(o, _sdpa(q, pos, k, v), rtol=1e-11, atol=1e-12)
    # lse: scipy logsumexp over the masked scores, scores by a plain matmul
    G = Hq // Hkv
    for h in range(Hq):
        s = q[:, h, :] @ k[:, h // G, :].T / math.sqrt(d)
        s = np.where(np.arange(N)[None, :] <= pos[:, None], s, -np.inf)
        np.testing.assert_allclose(lse[:, h], scipy.special.logsumexp(s, axis=1), rtol=1e-12)


def test_attention_rows_are_softmax_rows_summing_to_one():
    # V = identity rows (N <= d): O row h equals the softmax probability row
    rng = np.random.default_rng(7)
    N, Hq, Hkv, d = 24, 2, 1, 32
    q = rng.standard_normal((N, Hq, d))
    k = rng.standard_normal((N, Hkv, d))
    v = np.zeros((N, Hkv, d))
    v[np.arange(N), 0, np.arange(N)] = 1.0
    pos = np.arange(N)
    o, _ = oracle.attention(q, pos, k, v)
    np.testing.assert_allclose(o.sum(-1), 1.0, rtol=0, atol=1e-13)
    for h in range(Hq):
        s = q[:, h] @ k[:, 0].T / math.sqrt(d)
        s = np.where(np.arange(N)[None, :] <= pos[:, None], s, -np.inf)
        np.testing.assert_allclose(o[:, h, :N], scipy.special.softmax(s, axis=1), rtol=1e-12, atol=1e-15)


def test_attention_special_cases():
    rng = np.random.default_rng(8)
    N, Hq, Hkv, d = 30, 4, 2, 16
    k = rng.standard_normal((N, Hkv, d))
    # constant V: every row returns the constant
    u = rng.standard_normal(d)
    vc = np.broadcast_to(u, (N, Hkv, d)).copy()
    o, _ = oracle.attention(rng.standard_normal((N, Hq, d)), np.arange(N), k, vc)
    np.testing.assert_allclose(o, np.broadcast_to(u, o.shape), rtol=1e-13, atol=1e-13)
    # q = 0: uniform weights, O is the running mean of visible values
    v = rng.standard_normal((N, Hkv, d))
    o, lse = oracle.attention(np.zeros((N, Hq, d)), np.arange(N), k, v)
    G = Hq // Hkv
    for r in range(N):
        for h in range(Hq):
            np.testing.assert_allclose(o[r, h], v[: r + 1, h // G].mean(0), rtol=1e-12, atol=1e-14)
            assert abs(lse[r, h] - math.log(r + 1)) < 1e-13
    # row 0 sees only key 0
    o, _ = oracle.attention(rng.standard_normal((1, Hq, d)), [0], k, v)
    np.testing.assert_allclose(o[0], v[0][np.arange(Hq) // G], rtol=1e-14)
    # a row with no visible key
    o, lse = oracle.attention(rng.standard_normal((1, Hq, d)), [-1], k, v)
    assert np.all(o == 0) and np.all(np.isneginf(lse))


def test_gqa_equals_mha_with_repeated_kv_heads():
    rng = np.random.default_rng(9)
    N, Hq, Hkv, d = 19, 8, 2, 32
    q = rng.standard_normal((N, Hq, d))
    k = rng.standard_normal((N, Hkv, d))
    v = rng.standard_normal((N, Hkv, d))
    o_gqa, l_gqa = oracle.attention(q, np.arange(N), k, v)
    rep = np.repeat(np.arange(Hkv), Hq // Hkv)  # head h -> kv head h // G
    o_mha, l_mha = oracle.attention(q, np.arange(N), k[:, rep], v[:, rep])
    assert np.array_equal(o_gqa, o_mha) and np.array_equal(l_gqa, l_mha)


# ----------------------------------------------------------- Claim 1 etc ----

def _prep(seed, T, Hq, Hkv, d, pos):
    li = inputs.layer_inputs(seed, T, Hq, Hkv, d)
    dec = oracle.bf16_decode
    _, _, qb, kb = oracle.qk_prep(dec(li.q_pre), dec(li.k_pre), dec(li.q_norm_w),
                                  dec(li.k_norm_w), pos, 1e6, 1e-6)
    return dec(qb), dec(kb), dec(li.v)


def test_claim1_reuse_rows_equal_prefill_rows_exactly():
    """Claim 1 (Sec. 3.3): prefix keys are the same whether computed with or
    without the suffix, and the suffix rows of prefill(c||q) equal reuse(c, q)."""
    Hq, Hkv, d, L, n = 4, 1, 64, 256, 8
    q, k, v = _prep(0, L + n, Hq, Hkv, d, np.arange(L + n))
    o_pre, lse_pre = oracle.prefill(q, k, v)
    o_reu, lse_reu = oracle.reuse(q[L:], L, k, v)
    assert np.array_equal(o_pre[L:], o_reu) and np.array_equal(lse_pre[L:], lse_reu)
    # prefix rows do not depend on the suffix
    o_c, _ = oracle.prefill(q[:L], k[:L], v[:L])
    assert np.array_equal(o_pre[:L], o_c)
    # the cached prefix keys do not depend on the suffix either
    _, kc, _ = _prep(0, L + n, Hq, Hkv, d, np.arange(L + n))
    assert np.array_equal(kc[:L], k[:L])


def test_shifted_failure_mode_diverges():
    """Sec. 3.2: wrong position ids or a mask that omits the cached context
    reproduce the 'shifted' failure; both must give different rows."""
    Hq, Hkv, d, L, n = 4, 1, 64, 64, 8
    li = inputs.layer_inputs(1, L + n, Hq, Hkv, d)
    dec = oracle.bf16_decode
    args = (dec(li.q_norm_w), dec(li.k_norm_w))
    _, _, qb, kb = oracle.qk_prep(dec(li.q_pre), dec(li.k_pre), *args, np.arange(L + n), 1e6, 1e-6)
    q, k, v = dec(qb), dec(kb), dec(li.v)
    o_ok, _ = oracle.reuse(q[L:], L, k, v)
    # positions restarted at 0 for the continuation
    _, _, qs, ks = oracle.qk_prep(dec(li.q_pre[L:]), dec(li.k_pre[L:]), *args, np.arange(n), 1e6, 1e-6)
    k_sh = np.concatenate([k[:L], dec(ks)])
    o_sh, _ = oracle.reuse(dec(qs), L, k_sh, v)
    assert np.max(np.abs(o_sh - o_ok)) > 1e-2
    # mask covering only the continuation (cached context not attended)
    o_mask, _ = oracle.attention(q[L:], np.arange(n), k[L:], v[L:])
    assert np.max(np.abs(o_mask - o_ok)) > 1e-2


def test_qk_prep_is_norm_then_rope_then_one_rounding():
    Hq, Hkv, d, T = 4, 2, 64, 9
    li = inputs.layer_inputs(2, T, Hq, Hkv, d)
    dec = oracle.bf16_decode
    pos = np.array([0, 1, 2, 255, 256, 3773, 3774, 32767, 40000])
    qf, kf, qb, kb = oracle.qk_prep(dec(li.q_pre), dec(li.k_pre), dec(li.q_norm_w),
                                    dec(li.k_norm_w), pos, 1e6, 1e-6)
    want_q = _rope_complex(F.rms_norm(torch.from_numpy(dec(li.q_pre)), (d,),
                                      weight=torch.from_numpy(dec(li.q_norm_w)), eps=1e-6).numpy(),
                           pos[:, None], 1e6)
    np.testing.assert_allclose(qf, want_q, rtol=1e-10, atol=1e-11)
    # one rounding, to the nearest bf16 of the fp64 value (both q and k)
    for b, f in ((qb, qf), (kb, kf)):
        err = np.abs(dec(b) - f)
        ulp = 2.0 ** (np.floor(np.log2(np.abs(f))) - 7)
        assert np.all(err <= 0.5 * ulp * (1 + 1e-12))


# ----------------------------------------------------------- the paper's numbers ----

def test_artifact_size_matches_table1_and_sec5():
    s = {r[0]: float(r[1]) for r in read_golden("paper_scalars.txt")}
    per_tok = oracle.artifact_bytes(int(s["layers"]), int(s["kv_heads"]), int(s["head_dim"]), 1)
    assert per_tok == 147456
    assert abs(per_tok / 1e6 - s["mb_per_token"]) < 1.5e-3
    for row in read_golden("table1_cost.txt"):
        L, mb = int(row[0]), float(row[3])
        assert abs(oracle.artifact_bytes(36, 8, 128, L) / 1e6 - mb) <= 1.0
    fp16 = oracle.artifact_bytes(36, 8, 128, int(s["int8_probe_tokens"])) / 1e6
    assert abs(fp16 - s["int8_probe_fp16_mb"]) < 0.1
    assert abs(fp16 / 2 - s["int8_probe_int8_mb"]) < 0.1


def test_cost_model_reproduces_break_even_and_savings():
    s = {r[0]: float(r[1]) for r in read_golden("paper_scalars.txt")}
    rows = [(int(r[0]), float(r[1]), float(r[2]), float(r[4])) for r in read_golden("table1_cost.txt")]
    nstars = [oracle.break_even(cp, cr) for _, cp, cr, _ in rows]
    assert round(min(nstars), 2) == s["nstar_lo"] and round(max(nstars), 2) == s["nstar_hi"]
    for _, cp, cr, speed in rows:
        assert abs(cp / cr - speed) <= 0.1
        flat, reuse = oracle.per_call_cost(cp, cr, [1, 10, 1000])
        assert np.all(flat == cp) and reuse[0] == pytest.approx(cp + cr)
        assert reuse[2] == pytest.approx(cp / 1000 + cr)
    sav = {L: 1000 * (cp - cr) for L, cp, cr, _ in rows}
    assert abs(sav[255] - s["saving_n1000_255_s"]) / s["saving_n1000_255_s"] < 0.05
    assert abs(sav[3774] - s["saving_n1000_3774_s"]) / s["saving_n1000_3774_s"] < 0.05


# -------------------------------------------------------- int8 artifact ----
# Sec. 5 "Quantizing the artifact": per-tensor symmetric int8.

def _near_tie(x32, s):
    r = np.abs(x32.astype(np.float64) / np.float64(s))
    return np.abs(r - np.floor(r) - 0.5) < 1e-4


def test_q8_codes_match_torch_per_tensor_quantizer():
    """torch.quantize_per_tensor (symmetric: zero point 0) with the oracle's
    scale gives the same codes away from rounding ties."""
    x = inputs.normal_bf16(21, (8, 300, 64))
    codes, s = oracle.q8_quantize(x)
    x32 = oracle.bf16_decode(x).astype(np.float32)
    t = torch.quantize_per_tensor(torch.from_numpy(x32), float(s), 0, torch.qint8).int_repr().numpy()
    ok = ~_near_tie(x32, s)
    assert ok.mean() > 0.99
    assert np.array_equal(codes[ok], t[ok])
    assert s == np.float32(np.max(np.abs(x32)) / np.float32(127))


def test_q8_extremes_bound_and_brute_force():
    """The largest magnitude maps to +-127 (negative here); every code is the
    nearest multiple of s (brute force over all 255 codes); |code*s - x| <= s/2;
    the bf16 dequantised value adds at most half a bf16 ulp."""
    rng = np.random.default_rng(3)
    x32 = rng.standard_normal((4, 50, 16)).astype(np.float32)
    x32[1, 7, 3] = -9.5
    x = inputs.to_bf16_bits(x32)
    codes, s = oracle.q8_quantize(x)
    xv = oracle.bf16_decode(x)
    assert codes[1, 7, 3] == -127 and np.abs(codes).max() == 127
    cand = np.arange(-127, 128, dtype=np.float64) * np.float64(s)
    best = np.argmin(np.abs(xv.reshape(-1, 1) - cand[None, :]), axis=1) - 127
    ok = ~_near_tie(xv.astype(np.float32), s).reshape(-1)
    assert np.array_equal(codes.reshape(-1)[ok], best[ok])
    assert np.all(np.abs(codes * np.float64(s) - xv) <= 0.5 * s * (1 + 1e-5))
    deq = oracle.bf16_decode(oracle.q8_dequantize(codes, s))
    exact = codes * np.float64(s)
    ulp = 2.0 ** (np.floor(np.log2(np.maximum(np.abs(exact), 1e-30))) - 7)
    assert np.all(np.abs(deq - exact) <= 0.5 * ulp * (1 + 1e-6) + 1e-30)


def test_q8_invariants_symmetry_scaling_zero():
    """Symmetric: q(-x) = -q(x) with the same scale; a power-of-two factor
    scales s and leaves the codes; an all-zero tensor has s = 0, codes 0."""
    x32 = np.random.default_rng(4).standard_normal((3, 40, 32)).astype(np.float32)
    x = inputs.to_bf16_bits(x32)
    c, s = oracle.q8_quantize(x)
    cn, sn = oracle.q8_quantize(x ^ np.uint16(0x8000))
    assert sn == s and np.array_equal(cn, -c)
    c4, s4 = oracle.q8_quantize(inputs.to_bf16_bits(oracle.bf16_decode(x).astype(np.float32) * 4))
    assert s4 == 4 * s and np.array_equal(c4, c)
    cz, sz = oracle.q8_quantize(np.zeros((5, 8), dtype=np.uint16))
    assert sz == 0 and not cz.any()
    assert not oracle.q8_dequantize(cz, sz).any()


def test_q8_artifact_has_one_scale_per_layer_tensor():
    """Per tensor = one layer's K (or V) over all KV heads and positions: a
    large value in one head of layer 1's V moves only that tensor's scale, and
    every head of it."""
    art = inputs.normal_bf16(5, (3, 2, 4, 20, 16))
    sc, codes = oracle.q8_artifact(art)
    big = art.copy()
    big[1, 1, 2, 5, 7] = inputs.to_bf16_bits(np.array([40.0], dtype=np.float32))[0]
    sc2, codes2 = oracle.q8_artifact(big)
    changed = sc2 != sc
    assert changed[1, 1] and changed.sum() == 1
    assert sc2[1, 1] == np.float32(np.float32(40.0) / np.float32(127))
    assert codes2[1, 1, 2, 5, 7] == 127
    assert np.array_equal(codes2[0], codes[0]) and np.array_equal(codes2[2], codes[2])
    for l in range(3):
        for kv in range(2):
            c, s = oracle.q8_quantize(art[l, kv])
            assert s == sc[l, kv] and np.array_equal(c, codes[l, kv])
    back = oracle.q8_artifact_dequantize(sc, codes)
    xv = oracle.bf16_decode(art)
    err = np.abs(oracle.bf16_decode(back) - xv)
    # s/2 from the code, plus half a bf16 ulp of the dequantised value
    bound = sc.astype(np.float64)[:, :, None, None, None] * 0.5 * (1 + 1e-5) + (np.abs(xv) + sc.max()) * 2.0 ** -8
    assert np.all(err <= bound)


def test_q8_artifact_values_are_code_times_scale_within_the_quantisation_bound():
    """The exact dequantised tensors: within s/2 of the original values (round
    to nearest), one bf16 rounding away from q8_artifact_dequantize, the
    extreme element reproduced to the scale's rounding, zero for s = 0, and
    brute force for a few elements (code times scale in exact rationals)."""
    from fractions import Fraction
    art = inputs.normal_bf16(6, (2, 2, 3, 40, 16))
    art[1, 0] = 0
    sc, codes = oracle.q8_artifact(art)
    vals = oracle.q8_artifact_values(sc, codes)
    xv = oracle.bf16_decode(art)
    bound = sc.astype(np.float64)[:, :, None, None, None] * 0.5 * (1 + 1e-5)
    assert np.all(np.abs(vals - xv) <= bound)
    assert np.array_equal(oracle.bf16_encode(vals), oracle.q8_artifact_dequantize(sc, codes))
    assert not vals[1, 0].any()
    l, kv = 0, 1
    i = np.unravel_index(np.argmax(np.abs(xv[l, kv])), xv[l, kv].shape)
    assert abs(vals[l, kv][i] - xv[l, kv][i]) <= abs(xv[l, kv][i]) * 2.0 ** -23
    rng = np.random.default_rng(0)
    for _ in range(20):
        j = tuple(int(rng.integers(0, n)) for n in codes.shape)
        want = Fraction(int(codes[j])) * Fraction(float(sc[j[0], j[1]]))
        assert Fraction(float(vals[j])) == want


def test_q8_artifact_size_matches_sec5_probe():
    """Sec. 5: the 692-token artifact is 102.1 MB at 16 bits and 51.1 MB at int8 (2.0x)."""
    s = {r[0]: float(r[1]) for r in read_golden("paper_scalars.txt")}
    n = int(s["int8_probe_tokens"])
    q8 = oracle.q8_artifact_bytes(36, 8, 128, n)
    assert abs(q8 / 1e6 - s["int8_probe_int8_mb"]) < 0.1
    assert q8 == 288 + 36 * 2 * 8 * 128 * n
    assert round(oracle.artifact_bytes(36, 8, 128, n) / q8, 1) == 2.0


# ----------------------------------------------------------- full layer ----

def _layer_case(seed, T, P, hidden=96, inter=160, Hq=4, Hkv=2, d=32):
    rng = np.random.default_rng(seed)
    bits = inputs.to_bf16_bits

    def w(o, i):
        return bits((rng.standard_normal((o, i)) / np.sqrt(i)).astype(np.float32))

    def nw(n):
        return bits((1 + 0.1 * rng.standard_normal(n)).astype(np.float32))

    W = {"input_norm": nw(hidden), "wq": w(Hq * d, hidden), "wk": w(Hkv * d, hidden), "wv": w(Hkv * d, hidden),
         "q_norm": nw(d), "k_norm": nw(d), "wo": w(hidden, Hq * d), "post_norm": nw(hidden),
         "w_gate": w(inter, hidden), "w_up": w(inter, hidden), "w_down": w(hidden, inter)}
    h = bits(rng.standard_normal((P + T, hidden)).astype(np.float32))
    return W, h, dict(n_q_heads=Hq, n_kv_heads=Hkv, theta=1e6, eps=1e-6)


def _torch_layer(h_bits, W, pos, kc, vc, n_q_heads, n_kv_heads, theta, eps):
    """The same layer from torch's own routines (fp64, bf16 at each tensor
    boundary): F.rms_norm, F.linear, complex-exponential RoPE, SDPA with an
    explicit causal mask, F.silu."""
    def t(b):
        return torch.from_numpy(oracle.bf16_decode(b))

    def r(x):
        return x.to(torch.bfloat16).to(torch.float64)

    Hq, Hkv = n_q_heads, n_kv_heads
    d = W["q_norm"].shape[0]
    T = h_bits.shape[0]
    h = t(h_bits)
    x = r(F.rms_norm(h, (h.shape[1],), t(W["input_norm"]), eps))
    q = r(F.linear(x, t(W["wq"]))).view(T, Hq, d)
    k = r(F.linear(x, t(W["wk"]))).view(T, Hkv, d)
    v = r(F.linear(x, t(W["wv"]))).view(T, Hkv, d)

    def rope(y):
        ang = torch.from_numpy(np.asarray(pos, dtype=np.float64))[:, None] * theta ** (
            -torch.arange(d // 2, dtype=torch.float64) * 2 / d)
        z = torch.complex(y[..., : d // 2], y[..., d // 2:]) * torch.polar(torch.ones_like(ang), ang)[:, None, :]
        return torch.cat([z.real, z.imag], dim=-1)

    q = r(rope(F.rms_norm(q, (d,), t(W["q_norm"]), eps)))
    k = r(rope(F.rms_norm(k, (d,), t(W["k_norm"]), eps)))
    K = torch.cat([t(kc), k]).repeat_interleave(Hq // Hkv, dim=1)
    V = torch.cat([t(vc), v]).repeat_interleave(Hq // Hkv, dim=1)
    mask = torch.arange(K.shape[0])[None, :] <= torch.from_numpy(np.asarray(pos))[:, None]
    o = F.scaled_dot_product_attention(q.transpose(0, 1), K.transpose(0, 1), V.transpose(0, 1),
                                       attn_mask=mask[None]).transpose(0, 1)
    o = r(o)
    h1 = r(h + F.linear(o.reshape(T, Hq * d), t(W["wo"])))
    x2 = r(F.rms_norm(h1, (h1.shape[1],), t(W["post_norm"]), eps))
    a = r(F.silu(r(F.linear(x2, t(W["w_gate"])))) * r(F.linear(x2, t(W["w_up"]))))
    return r(h1 + F.linear(a, t(W["w_down"]))), o


def test_layer_matches_torch_composition():
    """The oracle's layer against torch's own norm / linear / SDPA / silu at the
    same bf16 boundaries: equal up to the rare bf16 rounding flip that a
    different fp64 summation order can cause."""
    T, P = 7, 9
    W, h, cfg = _layer_case(31, T, P)
    pos = np.arange(P, P + T)
    kc = inputs.normal_bf16(32, (P, cfg["n_kv_heads"], 32))
    vc = inputs.normal_bf16(33, (P, cfg["n_kv_heads"], 32))
    out, kb, vb, ob = oracle.layer_forward(h[P:], W, pos, kc, vc, **cfg)
    ref, oref = _torch_layer(h[P:], W, pos, kc, vc, **cfg)
    got = oracle.bf16_decode(out)
    assert np.mean(got == ref.numpy()) > 0.98
    assert np.linalg.norm(got - ref.numpy()) / np.linalg.norm(ref.numpy()) < 2e-3
    assert np.mean(oracle.bf16_decode(ob) == oref.numpy()) > 0.98


def test_layer_residual_identity_and_claim1():
    """Zero output and down projections leave the residual stream unchanged
    bit for bit; the layer over prefix||suffix equals the layer over the prefix
    then the suffix with the prefix's keys and values as the cache (Claim 1 at
    the layer), and earlier rows do not depend on later tokens."""
    T, P = 6, 10
    W, h, cfg = _layer_case(41, T, P)
    Z = dict(W)
    Z["wo"] = np.zeros_like(W["wo"])
    Z["w_down"] = np.zeros_like(W["w_down"])
    empty = np.zeros((0, cfg["n_kv_heads"], 32), dtype=np.uint16)
    out, _, _, _ = oracle.layer_forward(h, Z, np.arange(P + T), empty, empty, **cfg)
    assert np.array_equal(out, h)
    full, kf, vf, _ = oracle.layer_forward(h, W, np.arange(P + T), empty, empty, **cfg)
    pre, kp, vp, _ = oracle.layer_forward(h[:P], W, np.arange(P), empty, empty, **cfg)
    suf, ks, vs, _ = oracle.layer_forward(h[P:], W, np.arange(P, P + T), kp, vp, **cfg)
    assert np.array_equal(full[:P], pre) and np.array_equal(full[P:], suf)
    assert np.array_equal(kf, np.concatenate([kp, ks])) and np.array_equal(vf, np.concatenate([vp, vs]))


def test_layer_flops_by_count():
    """Closed form of layer_flops against a count of the multiply-adds of each
    GEMM and attention pair for a small case."""
    hidden, inter, Hq, Hkv, d, T, P = 96, 160, 4, 2, 32, 5, 11
    pairs = sum(P + t + 1 for t in range(T))
    macs = T * hidden * Hq * d + 2 * T * hidden * Hkv * d + T * Hq * d * hidden  # q, k, v, o
    macs += 3 * T * hidden * inter  # gate, up, down
    macs += 2 * Hq * d * pairs  # QK^T and PV per visible pair
    assert oracle.layer_flops(T, pairs, hidden, inter, Hq, Hkv, d) == 2 * macs


def test_linear_matches_torch_and_closed_forms():
    """The projection step against torch's F.linear in fp64 at the same bf16
    boundary (a transposed operand or a dropped residual fails it), the
    identity matrix (y = x), a zero matrix (y = c), and a single nonzero weight
    (y[:, n] = w x[:, k])."""
    T, N, K = 13, 24, 40
    x = inputs.normal_bf16(71, (T, K))
    w = inputs.normal_bf16(72, (N, K))
    c = inputs.normal_bf16(73, (T, N))
    t = lambda b: torch.from_numpy(oracle.bf16_decode(b))
    ref = F.linear(t(x), t(w)) + t(c)
    got = oracle.bf16_decode(oracle.linear(x, w, c))
    assert np.array_equal(got, t(oracle.bf16_encode(ref.numpy())).numpy())
    rt = ref.numpy()
    assert np.all(np.abs(got - rt) <= np.abs(rt) * 2.0 ** -8 + 1e-30)  # one rounding: half an ulp
    eye = oracle.bf16_encode(np.eye(K))
    assert np.array_equal(oracle.linear(x, eye), x)
    assert np.array_equal(oracle.linear(x, np.zeros((N, K), np.uint16), c), c)
    one = np.zeros((N, K))
    one[5, 7] = 2.0
    y = oracle.bf16_decode(oracle.linear(x, oracle.bf16_encode(one)))
    assert np.array_equal(y[:, 5], 2.0 * oracle.bf16_decode(x)[:, 7]) and not y[:, :5].any()


def test_linear_swiglu_matches_torch_composition():
    """The gate/up/SwiGLU steps against torch's F.silu(F.linear) * F.linear at
    the same bf16 boundaries; swapping gate and up (a plausible slip) differs."""
    T, I, K = 9, 16, 32
    x = inputs.normal_bf16(74, (T, K))
    wg = inputs.normal_bf16(75, (I, K))
    wu = inputs.normal_bf16(76, (I, K))
    t = lambda b: torch.from_numpy(oracle.bf16_decode(b))
    r = lambda v: t(oracle.bf16_encode(v.numpy()))
    ref = r(F.silu(r(F.linear(t(x), t(wg)))) * r(F.linear(t(x), t(wu))))
    got = oracle.bf16_decode(oracle.linear_swiglu(x, wg, wu))
    assert np.mean(got == ref.numpy()) > 0.99
    assert np.abs(got - ref.numpy()).max() <= 2.0 ** -7 * np.abs(ref.numpy()).max()
    swapped = oracle.bf16_decode(oracle.linear_swiglu(x, wu, wg))
    assert np.mean(swapped == got) < 0.5


# ------------------------------------------------------------ inputs ----

def test_inputs_are_seeded_and_shaped():
    a = inputs.layer_inputs(0, 8, 4, 1, 64)
    b = inputs.layer_inputs(0, 8, 4, 1, 64)
    assert a.q_pre.shape == (8, 4, 64) and a.k_pre.shape == (8, 1, 64) and a.v.shape == (8, 1, 64)
    assert np.array_equal(a.q_pre, b.q_pre) and np.array_equal(a.k_norm_w, b.k_norm_w)
    x = np.random.default_rng(0).standard_normal(1000).astype(np.float32)
    assert np.array_equal(inputs.to_bf16_bits(x), _torch_bf16_bits(x))
    lens = inputs.ragged_lengths(0, 256, 16, 512)
    assert lens.min() >= 16 and lens.max() <= 512
