"""GPU parity of the int8 artifact (Sec. 5 "Quantizing the artifact"): the
library's export against the oracle's codes and scales bit for bit, its load
against the oracle's dequantised cache bit for bit, reuse attention over an
int8-loaded prefix against the oracle over the dequantised keys and values,
and the argument checks of the int8 entry points."""
import numpy as np
import pytest

import oracle
from harness import Scenario, bits_of, check_close, f64_of, oracle_prep, tdev
from paper_2606_13361_gb300 import inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def kvr():
    from paper_2606_13361_gb300 import kvr as k
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return k


def _ctx(kvr, Hq, Hkv, d, layers=1, max_positions=8192, n_pages=64):
    return kvr.Context(kvr.make_desc(layers, Hq, Hkv, d, max_positions), n_pages, 16, 0)


def _status(kvr, C):
    st = kvr.kvr_sync_status(C.ctx)
    assert st == kvr.KVR_OK, kvr.kvr_last_error()


def q8_pack(scales: np.ndarray, codes: np.ndarray) -> np.ndarray:
    """The int8 artifact's byte layout: fp32 scales [layers][2] padded to 16
    bytes, then the codes [layers][2][Hkv][L][d]."""
    layers = scales.shape[0]
    pad = (8 * layers + 15) // 16 * 16
    buf = np.zeros(pad + codes.size, dtype=np.uint8)
    buf[: 8 * layers] = np.ascontiguousarray(scales, dtype="<f4").view(np.uint8).reshape(-1)
    buf[pad:] = np.ascontiguousarray(codes).view(np.uint8).reshape(-1)
    return buf


def q8_unpack(buf: np.ndarray, shape):
    layers = shape[0]
    pad = (8 * layers + 15) // 16 * 16
    scales = buf[: 8 * layers].view("<f4").reshape(layers, 2)
    return scales, buf[pad:].view(np.int8).reshape(shape)


def _host(t, where):
    if where == "device":
        return t.cuda(), True
    return t.cpu().pin_memory(), False


SHAPES = [(3, 8, 2, 128, 300), (1, 4, 1, 64, 129), (2, 32, 8, 128, 1000), (1, 4, 1, 128, 5)]


@pytest.mark.parametrize("where", ["device", "pinned"])
@pytest.mark.parametrize("layers,Hq,Hkv,d,L", SHAPES)
def test_q8_export_codes_and_scales_are_the_oracles(kvr, where, layers, Hq, Hkv, d, L):
    """Algorithm 1 with the Sec. 5 int8 artifact: same codes and scales as the
    oracle, bit for bit (the integer decision is an fp32 division on both sides),
    including an all-zero tensor (s = 0) and one with a large outlier."""
    C = _ctx(kvr, Hq, Hkv, d, layers=layers)
    art = inputs.normal_bf16(7, (layers, 2, Hkv, L, d))
    art[0, 1] = 0                                                       # s = 0
    art[-1, 0, Hkv - 1, L - 1, d - 1] = inputs.to_bf16_bits(np.array([-37.0], np.float32))[0]
    p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, 1, L), tdev(art), True)
    n = kvr.kvr_artifact_bytes_q8(C.desc, L)
    assert n == oracle.q8_artifact_bytes(layers, Hkv, d, L)
    out, on_dev = _host(torch.zeros(n, dtype=torch.uint8), where)
    meta = kvr.kvr_export_kv_q8(C.ctx, p, out, on_dev)
    torch.cuda.synchronize()
    _status(kvr, C)
    assert (meta.dtype, meta.L, meta.model_id) == (kvr.KVR_DTYPE_Q8, L, C.desc.model_id)
    scales, codes = q8_unpack(out.cpu().numpy(), art.shape)
    s_ref, c_ref = oracle.q8_artifact(art)
    assert np.array_equal(scales.view(np.uint32), s_ref.view(np.uint32))
    assert np.array_equal(codes, c_ref)
    assert scales[0, 1] == 0 and codes[-1, 0, Hkv - 1, L - 1, d - 1] == -127
    C.close()


@pytest.mark.parametrize("where", ["device", "pinned"])
@pytest.mark.parametrize("layers,Hq,Hkv,d,L", SHAPES)
def test_q8_load_is_the_oracles_dequantised_cache(kvr, where, layers, Hq, Hkv, d, L):
    """Algorithm 2 on an int8 artifact: the cache holds bf16(code * s) for every
    element, bit for bit against the oracle."""
    C = _ctx(kvr, Hq, Hkv, d, layers=layers)
    s_ref, c_ref = oracle.q8_artifact(inputs.normal_bf16(8, (layers, 2, Hkv, L, d)))
    src, on_dev = _host(torch.from_numpy(q8_pack(s_ref, c_ref)), where)
    p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, kvr.KVR_DTYPE_Q8, L), src, on_dev)
    assert kvr.kvr_seq_length(C.ctx, p) == L
    back = torch.empty(kvr.kvr_artifact_bytes(C.desc, L), dtype=torch.uint8, device="cuda")
    kvr.kvr_export_kv(C.ctx, p, back, True)
    _status(kvr, C)
    got = bits_of(back.view(torch.bfloat16)).reshape(c_ref.shape)
    assert np.array_equal(got, oracle.q8_artifact_dequantize(s_ref, c_ref))
    C.close()


@pytest.mark.parametrize("Hq,Hkv,d,L,qs", [(32, 8, 128, 3774, [64]), (32, 8, 128, 3774, [1]),
                                           (4, 1, 64, 700, [3, 130])])
def test_q8_reuse_attention_matches_oracle_and_differs_from_bf16(kvr, Hq, Hkv, d, L, qs):
    """Reuse over an int8-loaded prefix equals the oracle's attention over the
    dequantised prefix keys/values (within the tolerance) and is no longer
    bitwise the bf16 path's result (Sec. 5: int8 breaks exactness)."""
    sc = Scenario(9, Hq, Hkv, d, L, qs)
    C = _ctx(kvr, Hq, Hkv, d, n_pages=160)
    qb, kb = sc.oracle_prefix()
    v_pre = sc.li.v[:L]
    art = np.ascontiguousarray(np.stack([np.transpose(kb, (1, 0, 2)), np.transpose(v_pre, (1, 0, 2))])[None])
    s_ref, c_ref = oracle.q8_artifact(art)
    deq = oracle.q8_artifact_dequantize(s_ref, c_ref)
    outs = {}
    for kind in ("q8", "bf16"):
        if kind == "q8":
            p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, kvr.KVR_DTYPE_Q8, L),
                                torch.from_numpy(q8_pack(s_ref, c_ref)).cuda(), True)
        else:
            p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, 1, L), tdev(art), True)
        seqs = [kvr.kvr_seq_fork(C.ctx, p) for _ in qs]
        qp = np.concatenate([sc.li.q_pre[sc.suffix(b)] for b in range(len(qs))])
        kp = np.concatenate([sc.li.k_pre[sc.suffix(b)] for b in range(len(qs))])
        vv = np.concatenate([sc.li.v[sc.suffix(b)] for b in range(len(qs))])
        cu = np.concatenate([[0], np.cumsum(qs)]).astype(np.int64)
        q_out = torch.empty(qp.shape, dtype=torch.bfloat16, device="cuda")
        kvr.kvr_append_kv(C.ctx, 0, seqs, [L] * len(qs), cu, tdev(qp), tdev(kp), tdev(vv),
                          tdev(sc.li.q_norm_w), tdev(sc.li.k_norm_w), q_out)
        out = torch.empty_like(q_out)
        kvr.kvr_reuse_attn(C.ctx, 0, seqs, cu, q_out, out)
        _status(kvr, C)
        outs[kind] = f64_of(out)
    k_deq = np.transpose(deq[0, 0], (1, 0, 2))
    v_deq = np.transpose(deq[0, 1], (1, 0, 2))
    for b in range(len(qs)):
        o_ref, _ = _oracle_q8(sc, b, k_deq, v_deq)
        check_close(outs["q8"][cu[b]:cu[b + 1]], o_ref, f"int8 reuse consumer {b}")
    assert not np.array_equal(outs["q8"], outs["bf16"])
    C.close()


def _oracle_q8(sc, b, k_deq_bits, v_deq_bits):
    """Oracle reuse rows of consumer b over the dequantised prefix (bf16 bits
    [L][Hkv][d]) and its own exact suffix keys and values."""
    li = sc.li
    sl = sc.suffix(b)
    sub = inputs.LayerInputs(li.q_pre[sl], li.k_pre[sl], li.v[sl], li.q_norm_w, li.k_norm_w)
    n = sl.stop - sl.start
    qb, kb = oracle_prep(sub, sc.L + np.arange(n))
    dec = oracle.bf16_decode
    k_all = np.concatenate([dec(k_deq_bits), dec(kb)])
    v_all = np.concatenate([dec(v_deq_bits), dec(li.v[sl])])
    return oracle.reuse(dec(qb), sc.L, k_all, v_all)


def test_q8_entry_points_reject_bad_buffers(kvr):
    """Pageable host memory: UNSUPPORTED (no kernel reads it); a buffer that is
    not 16-byte aligned: INVALID_ARG; another model's int8 artifact:
    META_MISMATCH (Algorithm 2's assert); nothing is enqueued for any."""
    C = _ctx(kvr, 4, 1, 64)
    L = 10
    n = kvr.kvr_artifact_bytes_q8(C.desc, L)
    meta = kvr.kvr_artifact_meta(C.desc.model_id, kvr.KVR_DTYPE_Q8, L)
    pageable = np.zeros(n, dtype=np.uint8)
    dev = torch.zeros(n + 64, dtype=torch.uint8, device="cuda")
    for src, on_dev, status in ((pageable, False, kvr.KVR_ERR_UNSUPPORTED),
                                (dev[8:], True, kvr.KVR_ERR_INVALID_ARG)):
        with pytest.raises(kvr.KvrError) as e:
            kvr.kvr_load_kv(C.ctx, meta, src, on_dev)
        assert e.value.status == status
    with pytest.raises(kvr.KvrError) as e:
        kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id + 1, kvr.KVR_DTYPE_Q8, L), dev, True)
    assert e.value.status == kvr.KVR_ERR_META_MISMATCH
    p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, 1, L),
                        tdev(inputs.normal_bf16(1, (1, 2, 1, L, 64))), True)
    for dst, on_dev, status in ((pageable, False, kvr.KVR_ERR_UNSUPPORTED),
                                (dev[8:], True, kvr.KVR_ERR_INVALID_ARG)):
        with pytest.raises(kvr.KvrError) as e:
            kvr.kvr_export_kv_q8(C.ctx, p, dst, on_dev)
        assert e.value.status == status
    _status(kvr, C)
    C.close()


def test_q8_container_file_round_trip(kvr, tmp_path):
    """Export int8, write the container, read it into pinned memory, load:
    the cache equals the oracle's dequantisation of the exported codes."""
    layers, Hq, Hkv, d, L = 2, 8, 2, 128, 333
    C = _ctx(kvr, Hq, Hkv, d, layers=layers)
    art = inputs.normal_bf16(10, (layers, 2, Hkv, L, d))
    p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, 1, L), tdev(art), True)
    dev = torch.empty(kvr.kvr_artifact_bytes_q8(C.desc, L), dtype=torch.uint8, device="cuda")
    meta = kvr.kvr_export_kv_q8(C.ctx, p, dev, True)
    torch.cuda.synchronize()
    path = tmp_path / "prefix_q8.kvra"
    kvr.save_artifact(path, C.desc, meta, dev.cpu())
    pinned = torch.empty(dev.numel(), dtype=torch.uint8).pin_memory()
    m2, _ = kvr.read_artifact(path, C.desc, out=pinned)
    assert (m2.dtype, m2.L) == (kvr.KVR_DTYPE_Q8, L)
    p2 = kvr.kvr_load_kv(C.ctx, m2, pinned, False)
    back = torch.empty(kvr.kvr_artifact_bytes(C.desc, L), dtype=torch.uint8, device="cuda")
    kvr.kvr_export_kv(C.ctx, p2, back, True)
    _status(kvr, C)
    s_ref, c_ref = oracle.q8_artifact(art)
    got = bits_of(back.view(torch.bfloat16)).reshape(art.shape)
    assert np.array_equal(got, oracle.q8_artifact_dequantize(s_ref, c_ref))
    C.close()


@pytest.mark.parametrize("Hq,Hkv,d,L,qs,v_scale", [
    (32, 8, 128, 3774, [1], 1.0), (32, 8, 128, 300, [1, 1], 1.0), (4, 1, 64, 700, [1], 1.0),
    (32, 8, 128, 1000, [64], 1.0), (32, 8, 128, 1000, [1], 2.0 ** -10), (4, 1, 128, 520, [2], 2.0 ** 6),
    (4, 1, 64, 100, [1], 1.0), (32, 8, 128, 20000, [1], 1.0)])
def test_q8_resident_prefix_matches_the_oracle(kvr, Hq, Hkv, d, L, qs, v_scale):
    """kvr_load_kv_q8_resident keeps the codes of the full pages in HBM.  The
    decode path (<= 8 rows per KV head: the fused decode step and few-row
    reuse) reads them as code * s exactly: parity with the oracle over those
    values for the full pages and over the bf16 cache for the tail page.  The
    many-row path reads the bf16 cache: parity with the dequantised oracle.
    V scaled by powers of two (a tiny and a large scale) exercises the f16
    staging of the probabilities; outputs are compared after dividing by that
    factor (exact).  The extra pages return to the pool when the sequences
    close."""
    sc = Scenario(41, Hq, Hkv, d, L, qs)
    li = sc.li
    if v_scale != 1.0:
        sc.li = inputs.LayerInputs(li.q_pre, li.k_pre, inputs.to_bf16_bits(oracle.bf16_decode(li.v) * v_scale),
                                   li.q_norm_w, li.k_norm_w)
    C = _ctx(kvr, Hq, Hkv, d, max_positions=max(8192, L + 512), n_pages=4 * (L // 128 + 4))
    free0 = kvr.kvr_free_pages(C.ctx)
    _, kb = sc.oracle_prefix()
    art = np.ascontiguousarray(np.stack([np.transpose(kb, (1, 0, 2)), np.transpose(sc.li.v[:L], (1, 0, 2))])[None])
    s_ref, c_ref = oracle.q8_artifact(art)
    vals = oracle.q8_artifact_values(s_ref, c_ref)[0]
    deq = oracle.bf16_decode(oracle.q8_artifact_dequantize(s_ref, c_ref))[0]
    full = (L // 128) * 128
    T, G = sum(qs), Hq // Hkv
    few = T * G <= 8
    pref = np.concatenate([vals[:, :, :full], deq[:, :, full:]], axis=2) if few else deq
    k_pre, v_pre = (np.transpose(pref[kv], (1, 0, 2)) for kv in range(2))
    p = kvr.kvr_load_kv_q8_resident(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, kvr.KVR_DTYPE_Q8, L),
                                    torch.from_numpy(q8_pack(s_ref, c_ref)).cuda(), True)
    seqs = [kvr.kvr_seq_fork(C.ctx, p) for _ in qs]
    cu = np.concatenate([[0], np.cumsum(qs)]).astype(np.int64)
    qp, kp, vv = (np.concatenate([x[sc.suffix(b)] for b in range(len(qs))])
                  for x in (sc.li.q_pre, sc.li.k_pre, sc.li.v))
    args = (tdev(qp), tdev(kp), tdev(vv), tdev(sc.li.q_norm_w), tdev(sc.li.k_norm_w))
    q_out = torch.empty(qp.shape, dtype=torch.bfloat16, device="cuda")
    outs = []
    if few:
        o = torch.empty_like(q_out)
        kvr.kvr_decode_step(C.ctx, 0, seqs, [L] * len(qs), cu, *args, q_out, o)
        outs.append(o)
    else:
        kvr.kvr_append_kv(C.ctx, 0, seqs, [L] * len(qs), cu, *args, q_out)
    o = torch.empty_like(q_out)
    kvr.kvr_reuse_attn(C.ctx, 0, seqs, cu, q_out, o)
    outs.append(o)
    _status(kvr, C)
    for o in outs:
        got = f64_of(o)
        for b in range(len(qs)):
            o_ref, _ = _oracle_values(sc, b, k_pre, v_pre)
            check_close(got[cu[b]:cu[b + 1]] / v_scale, o_ref / v_scale, f"int8-resident consumer {b}")
    for x in seqs + [p]:
        kvr.kvr_seq_close(C.ctx, x)
    assert kvr.kvr_free_pages(C.ctx) == free0
    C.close()


def _oracle_values(sc, b, k_prefix, v_prefix):
    """Oracle reuse rows of consumer b over prefix keys and values given as
    fp64 [L][Hkv][d] and its own exact suffix keys and values."""
    li = sc.li
    sl = sc.suffix(b)
    sub = inputs.LayerInputs(li.q_pre[sl], li.k_pre[sl], li.v[sl], li.q_norm_w, li.k_norm_w)
    n = sl.stop - sl.start
    qb, kb = oracle_prep(sub, sc.L + np.arange(n))
    dec = oracle.bf16_decode
    return oracle.reuse(dec(qb), sc.L, np.concatenate([k_prefix, dec(kb)]), np.concatenate([v_prefix, dec(li.v[sl])]))


def test_q8_resident_rejects_bad_requests(kvr):
    C = _ctx(kvr, 4, 1, 64)
    art = tdev(inputs.normal_bf16(1, (1, 2, 1, 200, 64)))
    with pytest.raises(kvr.KvrError) as e:  # a bf16 artifact
        kvr.kvr_load_kv_q8_resident(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, 1, 200), art, True)
    assert e.value.status == kvr.KVR_ERR_INVALID_ARG
    with pytest.raises(kvr.KvrError) as e:  # another model
        kvr.kvr_load_kv_q8_resident(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id + 1, kvr.KVR_DTYPE_Q8, 200), art,
                                    True)
    assert e.value.status == kvr.KVR_ERR_META_MISMATCH
    _status(kvr, C)
    C.close()
