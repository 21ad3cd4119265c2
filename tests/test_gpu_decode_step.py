"""kvr_decode_step (Algorithm 2's per-layer step: append the new tokens, then
attend over the cached context) against the two separate calls it stands for
(bitwise: output, lse, roped q and the cache) and against the fp64 oracle."""
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
    assert torch.cuda.is_available()
    return k


def _inputs(li, sl_list):
    qp = np.concatenate([li.q_pre[s] for s in sl_list])
    kp = np.concatenate([li.k_pre[s] for s in sl_list])
    vv = np.concatenate([li.v[s] for s in sl_list])
    return tdev(qp), tdev(kp), tdev(vv)


def _export(kvr, C, seq):
    n = kvr.kvr_seq_length(C.ctx, seq)
    art = torch.empty(kvr.kvr_artifact_bytes(C.desc, n), dtype=torch.uint8, device="cuda")
    kvr.kvr_export_kv(C.ctx, seq, art, True)
    return bits_of(art.view(torch.bfloat16))


@pytest.mark.parametrize("Hq,Hkv,d,L,qs", [
    (32, 8, 128, 3774, [1]),        # the Qwen3-4B layer decode step
    (32, 8, 128, 1000, [1, 1]),     # two consumers of one prefix
    (4, 1, 64, 256, [1]),           # tiny layer, d = 64
    (8, 8, 128, 300, [1] * 8),      # MHA, eight consumers
    (32, 8, 128, 3774, [2]),        # two new tokens
    (32, 8, 128, 1000, [5, 3]),     # 32 rows per KV head: falls back to append + reuse
    (32, 8, 128, 127, [1]),         # new key opens a page
    (32, 8, 128, 384, [1]),         # 13 units of 32 keys per KV head: the first 6-warp count (8 CTAs)
    (32, 8, 128, 1536, [1]),        # 49 units: 9 CTAs of 6 warps, one pass
    (32, 8, 128, 2303, [1]),        # 72 units: 12 CTAs, the last single pass
    (32, 8, 128, 2304, [1]),        # 73 units: the first second pass of the 6-warp CTAs
    (32, 8, 128, 4607, [1]),        # 144 units: the last 6-warp count
    (32, 8, 128, 4608, [1]),        # 145 units: back to the 12-warp CTAs
])
def test_decode_step_equals_append_then_reuse(kvr, Hq, Hkv, d, L, qs):
    sc = Scenario(6, Hq, Hkv, d, L, qs)
    dec = oracle.bf16_decode
    outs = {}
    for mode in ("fused", "separate"):
        C = kvr.Context(kvr.make_desc(1, Hq, Hkv, d, 8192), n_pages=96, max_seqs=32)
        art = inputs.normal_bf16(7, (1, 2, Hkv, L, d))
        p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, 1, L), tdev(art), True)
        seqs = [kvr.kvr_seq_fork(C.ctx, p) for _ in qs]
        cu = np.concatenate([[0], np.cumsum(qs)]).astype(np.int64)
        qp, kp, vv = _inputs(sc.li, [sc.suffix(b) for b in range(len(qs))])
        T = int(cu[-1])
        q_out = torch.empty((T, Hq, d), dtype=torch.bfloat16, device="cuda")
        out = torch.empty_like(q_out)
        lse = torch.empty((T, Hq), dtype=torch.float32, device="cuda")
        w = (tdev(sc.li.q_norm_w), tdev(sc.li.k_norm_w))
        if mode == "fused":
            kvr.kvr_decode_step(C.ctx, 0, seqs, [L] * len(qs), cu, qp, kp, vv, *w, q_out, out, lse)
        else:
            kvr.kvr_append_kv(C.ctx, 0, seqs, [L] * len(qs), cu, qp, kp, vv, *w, q_out)
            kvr.kvr_reuse_attn(C.ctx, 0, seqs, cu, q_out, out, lse)
        kvr.kvr_seq_advance(C.ctx, seqs, qs)
        assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK, kvr.kvr_last_error()
        outs[mode] = (bits_of(out), lse.cpu().numpy(), bits_of(q_out), [_export(kvr, C, s) for s in seqs])
        C.close()
    f, s_ = outs["fused"], outs["separate"]
    assert np.array_equal(f[0], s_[0]) and np.array_equal(f[1], s_[1]) and np.array_equal(f[2], s_[2])
    for a, b in zip(f[3], s_[3]):
        assert np.array_equal(a, b)
    # and against the oracle (prefix = the stand-in artifact, suffix through the oracle's append)
    art = inputs.normal_bf16(7, (1, 2, Hkv, L, d))
    kpre = np.transpose(art[0, 0], (1, 0, 2))
    vpre = np.transpose(art[0, 1], (1, 0, 2))
    got = dec(f[0])
    for b in range(len(qs)):
        sl = sc.suffix(b)
        sub = inputs.LayerInputs(sc.li.q_pre[sl], sc.li.k_pre[sl], sc.li.v[sl], sc.li.q_norm_w, sc.li.k_norm_w)
        qb, kb = oracle_prep(sub, L + np.arange(qs[b]))
        o_ref, _ = oracle.reuse(dec(qb), L, np.concatenate([dec(kpre), dec(kb)]),
                                np.concatenate([dec(vpre), dec(sc.li.v[sl])]))
        check_close(got[cu[b]:cu[b + 1]], o_ref, f"decode step consumer {b}")


def test_decode_step_loop_matches_oracle(kvr):
    """24 decode steps of one consumer after a 3774-token document: every step's
    output against the oracle, which follows the same tokens."""
    Hq, Hkv, d, L, steps = 32, 8, 128, 3774, 24
    li = inputs.layer_inputs(8, L + steps, Hq, Hkv, d)
    dec = oracle.bf16_decode
    C = kvr.Context(kvr.make_desc(1, Hq, Hkv, d, 8192), n_pages=96, max_seqs=8)
    pre = inputs.LayerInputs(li.q_pre[:L], li.k_pre[:L], li.v[:L], li.q_norm_w, li.k_norm_w)
    _, kb = oracle_prep(pre, np.arange(L))
    art = np.ascontiguousarray(np.stack([np.transpose(kb, (1, 0, 2)), np.transpose(li.v[:L], (1, 0, 2))])[None])
    p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, 1, L), tdev(art), True)
    c = kvr.kvr_seq_fork(C.ctx, p)
    K, V = list(dec(kb)), list(dec(li.v[:L]))
    w = (tdev(li.q_norm_w), tdev(li.k_norm_w))
    out = torch.empty((1, Hq, d), dtype=torch.bfloat16, device="cuda")
    for t in range(steps):
        sl = slice(L + t, L + t + 1)
        kvr.kvr_decode_step(C.ctx, 0, [c], [L + t], [0, 1], tdev(li.q_pre[sl]), tdev(li.k_pre[sl]),
                            tdev(li.v[sl]), *w, None, out)
        kvr.kvr_seq_advance(C.ctx, [c], [1])
        sub = inputs.LayerInputs(li.q_pre[sl], li.k_pre[sl], li.v[sl], li.q_norm_w, li.k_norm_w)
        qn, kn = oracle_prep(sub, [L + t])
        K.append(dec(kn)[0])
        V.append(dec(li.v[sl])[0])
        o_ref, _ = oracle.attention(dec(qn), [L + t], np.stack(K), np.stack(V))
        check_close(f64_of(out), o_ref, f"decode step {t}")
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK
    C.close()


def test_decode_step_refuses_shifted_positions(kvr):
    C = kvr.Context(kvr.make_desc(1, 4, 1, 64, 4096), n_pages=8, max_seqs=4)
    s = kvr.kvr_seq_open(C.ctx)
    x = torch.zeros((1, 4, 64), dtype=torch.bfloat16, device="cuda")
    kv = torch.zeros((1, 1, 64), dtype=torch.bfloat16, device="cuda")
    w = torch.ones(64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(kvr.KvrError) as e:
        kvr.kvr_decode_step(C.ctx, 0, [s], [3], [0, 1], x, kv, kv, w, w, None, torch.empty_like(x))
    assert e.value.status == kvr.KVR_ERR_POSITION
    C.close()


@pytest.mark.parametrize("Hq,Hkv,d,L,qs", [
    (32, 8, 128, 20000, [1]),       # 626 units per KV head: more splits than one cluster holds
    (32, 8, 128, 33000, [1, 1]),    # two consumers of a 33K document
    (4, 1, 64, 14000, [2]),         # one KV head, d = 64
    (8, 8, 128, 12000, [1] * 8),    # MHA, eight consumers: 8 rows per KV head across the clusters
])
def test_long_context_decode_spans_clusters(kvr, Hq, Hkv, d, L, qs):
    """Decode-sized attention over long contexts, where a KV head's splits span
    several thread-block clusters and the last cluster to finish merges the
    partials: the fused step and the separate calls against the fp64 oracle,
    and repeated calls over the same cache bit for bit (the merge order does
    not depend on which cluster arrives last, and the arrival counts reset)."""
    dec = oracle.bf16_decode
    C = kvr.Context(kvr.make_desc(1, Hq, Hkv, d, L + 256), n_pages=2 * (L // 128) + 16, max_seqs=16)
    art = inputs.normal_bf16(17, (1, 2, Hkv, L, d))
    p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, 1, L), tdev(art), True)
    seqs = [kvr.kvr_seq_fork(C.ctx, p) for _ in qs]
    cu = np.concatenate([[0], np.cumsum(qs)]).astype(np.int64)
    T = int(cu[-1])
    li = inputs.layer_inputs(18, T, Hq, Hkv, d)
    w = (tdev(li.q_norm_w), tdev(li.k_norm_w))
    q_out = torch.empty((T, Hq, d), dtype=torch.bfloat16, device="cuda")
    out = torch.empty_like(q_out)
    kvr.kvr_decode_step(C.ctx, 0, seqs, [L] * len(qs), cu, tdev(li.q_pre), tdev(li.k_pre), tdev(li.v), *w,
                        q_out, out)
    again = []
    for _ in range(3):
        o2 = torch.empty_like(out)
        kvr.kvr_reuse_attn(C.ctx, 0, seqs, cu, q_out, o2)
        again.append(bits_of(o2))
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK, kvr.kvr_last_error()
    first = bits_of(out)
    for x in again:
        assert np.array_equal(x, first)
    kpre = dec(np.transpose(art[0, 0], (1, 0, 2)))
    vpre = dec(np.transpose(art[0, 1], (1, 0, 2)))
    got = dec(first)
    for b in range(len(qs)):
        sl = slice(int(cu[b]), int(cu[b + 1]))
        sub = inputs.LayerInputs(li.q_pre[sl], li.k_pre[sl], li.v[sl], li.q_norm_w, li.k_norm_w)
        qb, kb = oracle_prep(sub, L + np.arange(qs[b]))
        o_ref, _ = oracle.reuse(dec(qb), L, np.concatenate([kpre, dec(kb)]), np.concatenate([vpre, dec(li.v[sl])]))
        check_close(got[sl], o_ref, f"long-context decode consumer {b}")
    C.close()
