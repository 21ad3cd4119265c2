"""Parity at the workload sizes the benchmarks use (sampled rows against the
fp64 oracle; rows are independent, so a sample checks the launch as run):

  - shared-prefix serving: a 3774-token document, 64 consumers x 128 tokens,
    one reuse call per layer;
  - length sweep: L in {1K .. 32K}, prefill over L, reuse with q = 64 and a
    decode step, Qwen3-4B layer shapes;
  - hot document: L = 32768, 256 consumers with suffixes uniform in [16, 512],
    then decode steps of all 256 consumers together.

The cache holds two layers and the second (layer 1) is checked, so layer
addressing is exercised; the attention of every layer runs the same code."""
import numpy as np
import pytest

import oracle
from harness import check_close, f64_of, oracle_prep, tdev
from paper_2606_13361_gb300 import inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
HQ, HKV, D = 32, 8, 128
LAYER = 1


@pytest.fixture(scope="module")
def kvr():
    from paper_2606_13361_gb300 import kvr as k
    assert torch.cuda.is_available()
    return k


def _prefix(kvr, C, L, seed):
    """Document of L tokens through the oracle's append step; loaded into layer 1
    (layer 0 gets the same bytes).  Returns (prefix seq, k bf16 [L,Hkv,d], v bf16)."""
    li = inputs.layer_inputs(seed, L, HQ, HKV, D)
    _, kb = oracle_prep(li, np.arange(L))
    kv = np.stack([np.transpose(kb, (1, 0, 2)), np.transpose(li.v, (1, 0, 2))])
    art = np.ascontiguousarray(np.stack([kv, kv]))  # [layers=2][2][Hkv][L][d]
    p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, 1, L), tdev(art), True)
    return p, kb, li.v, li.q_norm_w, li.k_norm_w


def _append_batch(kvr, C, seqs, starts, tok_inputs, wq, wk):
    qp = np.concatenate([t.q_pre for t in tok_inputs])
    kp = np.concatenate([t.k_pre for t in tok_inputs])
    vv = np.concatenate([t.v for t in tok_inputs])
    cu = np.concatenate([[0], np.cumsum([t.q_pre.shape[0] for t in tok_inputs])]).astype(np.int64)
    q_out = torch.empty(qp.shape, dtype=torch.bfloat16, device="cuda")
    kvr.kvr_append_kv(C.ctx, LAYER, seqs, starts, cu, tdev(qp), tdev(kp), tdev(vv), tdev(wq), tdev(wk), q_out)
    return q_out, cu


def _oracle_rows(kpre, vpre, suffix_li, L, rows, wq, wk):
    dec = oracle.bf16_decode
    sub = inputs.LayerInputs(suffix_li.q_pre, suffix_li.k_pre, suffix_li.v, wq, wk)
    n = suffix_li.q_pre.shape[0]
    qb, kb = oracle_prep(sub, L + np.arange(n))
    o, _ = oracle.reuse(dec(qb), L, np.concatenate([dec(kpre), dec(kb)]),
                        np.concatenate([dec(vpre), dec(suffix_li.v)]), rows=rows)
    return o


def _tok_inputs(seed, n, wq, wk):
    li = inputs.layer_inputs(seed, n, HQ, HKV, D)
    return inputs.LayerInputs(li.q_pre, li.k_pre, li.v, wq, wk)


def test_shared_prefix_serving_64_consumers(kvr):
    L, B, q = 3774, 64, 128
    C = kvr.Context(kvr.make_desc(2, HQ, HKV, D, 8192), n_pages=200, max_seqs=B + 4)
    p, kpre, vpre, wq, wk = _prefix(kvr, C, L, seed=30)
    seqs = [kvr.kvr_seq_fork(C.ctx, p) for _ in range(B)]
    toks = [_tok_inputs(1000 + b, q, wq, wk) for b in range(B)]
    q_out, cu = _append_batch(kvr, C, seqs, [L] * B, toks, wq, wk)
    out = torch.empty_like(q_out)
    kvr.kvr_reuse_attn(C.ctx, LAYER, seqs, cu, q_out, out)
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK, kvr.kvr_last_error()
    got = f64_of(out)
    rows = np.array([0, 1, 31, 32, 63, 127])
    for b in (0, 1, 17, 40, 63):
        o_ref = _oracle_rows(kpre, vpre, toks[b], L, rows, wq, wk)
        check_close(got[cu[b] + rows], o_ref, f"serving consumer {b}")
    C.close()


@pytest.mark.parametrize("L", inputs.SWEEP_L)
def test_length_sweep_prefill_reuse_decode(kvr, L):
    q = 64
    C = kvr.Context(kvr.make_desc(2, HQ, HKV, D, 33000), n_pages=2 * (L // 128) + 16, max_seqs=8)
    # prefill over L through the GPU append, sampled rows
    li = inputs.layer_inputs(40, L, HQ, HKV, D)
    x = kvr.kvr_seq_open(C.ctx)
    qx, _ = _append_batch(kvr, C, [x], [0], [li], li.q_norm_w, li.k_norm_w)
    ox = torch.empty_like(qx)
    kvr.kvr_prefill_attn(C.ctx, LAYER, x, L, qx, ox)
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK, kvr.kvr_last_error()
    rng = np.random.default_rng(L)
    rows = np.unique(np.concatenate([[0, 127, 128, L - 1], rng.integers(0, L, 12)]))
    dec = oracle.bf16_decode
    qb, kb = oracle_prep(li, np.arange(L))
    o_ref, _ = oracle.prefill(dec(qb), dec(kb), dec(li.v), rows=rows)
    check_close(f64_of(ox)[rows], o_ref, f"prefill L={L}")
    kvr.kvr_seq_close(C.ctx, x)
    del qx, ox
    # reuse q = 64 after a loaded document of L tokens, then one decode step
    p, kpre, vpre, wq, wk = _prefix(kvr, C, L, seed=41)
    c = kvr.kvr_seq_fork(C.ctx, p)
    suf = _tok_inputs(42, q + 1, wq, wk)
    first = inputs.LayerInputs(suf.q_pre[:q], suf.k_pre[:q], suf.v[:q], wq, wk)
    qs, cu = _append_batch(kvr, C, [c], [L], [first], wq, wk)
    os_ = torch.empty_like(qs)
    kvr.kvr_reuse_attn(C.ctx, LAYER, [c], cu, qs, os_)
    kvr.kvr_seq_advance(C.ctx, [c], [q])
    od = torch.empty((1, HQ, D), dtype=torch.bfloat16, device="cuda")
    kvr.kvr_decode_step(C.ctx, LAYER, [c], [L + q], [0, 1], tdev(suf.q_pre[q:]), tdev(suf.k_pre[q:]),
                        tdev(suf.v[q:]), tdev(wq), tdev(wk), None, od)
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK, kvr.kvr_last_error()
    rows = np.array([0, 1, 31, 63, 64])
    o_ref = _oracle_rows(kpre, vpre, suf, L, rows, wq, wk)
    got = np.concatenate([f64_of(os_)[rows[:-1]], f64_of(od)])
    check_close(got, o_ref, f"reuse/decode L={L}")
    C.close()


def test_hot_document_256_consumers(kvr):
    L, B, steps = 32768, 256, 2
    qs = inputs.ragged_lengths(0, B, 16, 512)
    total = int(qs.sum())
    C = kvr.Context(kvr.make_desc(2, HQ, HKV, D, 33500), n_pages=256 + B * 7 + 8, max_seqs=B + 4)
    p, kpre, vpre, wq, wk = _prefix(kvr, C, L, seed=50)
    seqs = [kvr.kvr_seq_fork(C.ctx, p) for _ in range(B)]
    allt = inputs.layer_inputs(51, total + B * steps, HQ, HKV, D)
    cu = np.concatenate([[0], np.cumsum(qs)]).astype(np.int64)

    def consumer(b):
        sl = slice(int(cu[b]), int(cu[b + 1]))
        return inputs.LayerInputs(allt.q_pre[sl], allt.k_pre[sl], allt.v[sl], wq, wk)

    q_out, cu2 = _append_batch(kvr, C, seqs, [L] * B, [consumer(b) for b in range(B)], wq, wk)
    assert np.array_equal(cu, cu2)
    out = torch.empty_like(q_out)
    kvr.kvr_reuse_attn(C.ctx, LAYER, seqs, cu, q_out, out)
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK, kvr.kvr_last_error()
    got = f64_of(out)
    sample = (0, 5, 100, 255)
    for b in sample:
        rows = np.array(sorted({0, int(qs[b]) // 2, int(qs[b]) - 1}))
        o_ref = _oracle_rows(kpre, vpre, consumer(b), L, rows, wq, wk)
        check_close(got[cu[b] + rows], o_ref, f"hot document consumer {b}")
    kvr.kvr_seq_advance(C.ctx, seqs, [int(x) for x in qs])
    # decode steps of all 256 consumers together (shared prefix, one token each)
    hist = {b: consumer(b) for b in sample}
    for t in range(steps):
        sl = slice(total + t * B, total + (t + 1) * B)
        tok = inputs.LayerInputs(allt.q_pre[sl], allt.k_pre[sl], allt.v[sl], wq, wk)
        starts = [L + int(qs[b]) + t for b in range(B)]
        od = torch.empty((B, HQ, D), dtype=torch.bfloat16, device="cuda")
        qd = torch.empty_like(od)
        kvr.kvr_decode_step(C.ctx, LAYER, seqs, starts, list(range(B + 1)), tdev(tok.q_pre), tdev(tok.k_pre),
                            tdev(tok.v), tdev(wq), tdev(wk), qd, od)
        kvr.kvr_seq_advance(C.ctx, seqs, [1] * B)
        assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK, kvr.kvr_last_error()
        gd = f64_of(od)
        for b in sample:
            h = hist[b]
            hist[b] = inputs.LayerInputs(np.concatenate([h.q_pre, tok.q_pre[b:b + 1]]),
                                         np.concatenate([h.k_pre, tok.k_pre[b:b + 1]]),
                                         np.concatenate([h.v, tok.v[b:b + 1]]), wq, wk)
            n = hist[b].q_pre.shape[0]
            o_ref = _oracle_rows(kpre, vpre, hist[b], L, np.array([n - 1]), wq, wk)
            check_close(gd[b:b + 1], o_ref, f"hot document decode step {t} consumer {b}")
    C.close()
