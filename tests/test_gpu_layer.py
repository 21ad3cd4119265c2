"""GPU parity of the whole decoder layer (kvr_layer_forward) against the
oracle's layer (fp64 per operation, bf16 at every tensor boundary): prefill
from scratch over L tokens, then a reuse step of ragged suffixes over the
loaded prefix and a decode step, two layers deep, at a small shape and at the
Qwen3-4B layer shape."""
import numpy as np
import pytest

import oracle
from harness import bits_of, tdev
from paper_2606_13361_gb300 import inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

THETA, EPS = 1e6, 1e-6


@pytest.fixture(scope="module")
def kvr():
    from paper_2606_13361_gb300 import kvr as k
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return k


def make_weights(seed, hidden, inter, Hq, Hkv, d):
    """Random layer weights, bf16 bits: projections N(0, 1/fan_in), norm
    weights 1 + 0.1 N(0, 1)."""
    rng = np.random.default_rng(seed)
    bits = inputs.to_bf16_bits

    def w(o, i):
        return bits((rng.standard_normal((o, i)) / np.sqrt(i)).astype(np.float32))

    def nw(n):
        return bits((1 + 0.1 * rng.standard_normal(n)).astype(np.float32))

    return {"input_norm": nw(hidden), "wq": w(Hq * d, hidden), "wk": w(Hkv * d, hidden), "wv": w(Hkv * d, hidden),
            "q_norm": nw(d), "k_norm": nw(d), "wo": w(hidden, Hq * d), "post_norm": nw(hidden),
            "w_gate": w(inter, hidden), "w_up": w(inter, hidden), "w_down": w(hidden, inter)}


def device_weights(kvr, W):
    dev = {k: tdev(v) for k, v in W.items() if k not in ("w_gate", "w_up")}
    dev["w_gate_up"] = tdev(np.concatenate([W["w_gate"], W["w_up"]]))
    return dev, kvr.layer_weights(dev)


def check_layer(got_bits, want_bits, what, depth=1):
    """Layer outputs.  The GPU and the oracle round the same tensors to bf16;
    up to the attention they agree almost bit for bit (checked on the cache
    below), but the attention output carries the attention kernel's own error
    (bf16 P, fp32 sums: within the attention tolerance's 5e-3 relative RMS), and every
    element it moves shifts the output projection and the MLP after it.  The
    bound is that budget per layer of depth, and a max error of a few bf16
    ulps of the largest output."""
    g = oracle.bf16_decode(got_bits)
    w = oracle.bf16_decode(want_bits)
    rel = np.linalg.norm(g - w) / np.linalg.norm(w)
    mx = np.abs(g - w).max()
    ulp = 2.0 ** (np.floor(np.log2(np.abs(w).max())) - 7)
    print(f"{what}: rel {rel:.2e} max {mx:.2e} ({mx / ulp:.1f} ulp) bitwise {np.mean(got_bits == want_bits):.3f}")
    assert rel <= 5e-3 * depth and mx <= 4 * ulp, f"{what}: rel {rel:.2e} max {mx:.2e}"


def run_case(kvr, layers, hidden, inter, Hq, Hkv, d, L, qs):
    desc = kvr.make_desc(layers, Hq, Hkv, d, max_positions=L + max(qs) + 256)
    ld = kvr.kvr_layer_desc(hidden, inter)
    C = kvr.Context(desc, n_pages=4 * ((L + max(qs)) // 128 + 4), max_seqs=16)
    Ws = [make_weights(100 + l, hidden, inter, Hq, Hkv, d) for l in range(layers)]
    devs = [device_weights(kvr, W) for W in Ws]
    T_max = max(L, sum(qs) + len(qs))
    ws = torch.empty(kvr.kvr_layer_workspace_bytes(desc, ld, T_max), dtype=torch.uint8, device="cuda")
    h0 = inputs.normal_bf16(7, (L, hidden))
    # ---- prefill from scratch (Table 1 cost (a)) on the GPU and in the oracle
    x = kvr.kvr_seq_open(C.ctx)
    h = tdev(h0)
    for l in range(layers):
        nxt = torch.empty_like(h)
        kvr.kvr_layer_forward(C.ctx, l, ld, devs[l][1], [x], [0], [0, L], h, nxt, ws)
        h = nxt
    kvr.kvr_seq_advance(C.ctx, [x], [L])
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK, kvr.kvr_last_error()
    empty = np.zeros((0, Hkv, d), dtype=np.uint16)
    ho, caches = h0, []
    for l in range(layers):
        ho, kb, vb, _ = oracle.layer_forward(ho, Ws[l], np.arange(L), empty, empty, Hq, Hkv, THETA, EPS)
        caches.append((kb, vb))
    check_layer(bits_of(h), ho, "prefill", layers)
    # layer 0's cached keys and values depend only on the input: norm,
    # projection, QK-norm + RoPE -- no attention error in them yet
    art0 = torch.empty(kvr.kvr_artifact_bytes(desc, L), dtype=torch.uint8, device="cuda")
    kvr.kvr_export_kv(C.ctx, x, art0, True)
    a0 = bits_of(art0.view(torch.bfloat16)).reshape(layers, 2, Hkv, L, d)
    for kv, want in ((0, caches[0][0]), (1, caches[0][1])):
        got = np.transpose(a0[0, kv], (1, 0, 2))
        gd, wd = oracle.bf16_decode(got), oracle.bf16_decode(want)
        # ulp of each head vector's largest element: RoPE mixes pairs, so a
        # one-ulp flip of an input shows up in small outputs as many of their ulps
        ulp = 2.0 ** (np.floor(np.log2(np.abs(wd).max(axis=-1, keepdims=True))) - 7)
        print(f"layer-0 cache {kv}: bitwise {np.mean(got == want):.4f}, max {np.max(np.abs(gd - wd) / ulp):.2f} ulp")
        assert np.mean(got == want) >= 0.99 and np.all(np.abs(gd - wd) <= 3 * ulp), f"layer-0 cache {kv}"
    # ---- the artifact of the prefill, loaded, forked by the consumers (cost (b))
    art = torch.empty(kvr.kvr_artifact_bytes(desc, L), dtype=torch.uint8, device="cuda")
    p = kvr.kvr_load_kv(C.ctx, kvr.kvr_export_kv(C.ctx, x, art, True), art, True)
    seqs = [kvr.kvr_seq_fork(C.ctx, p) for _ in qs]
    cu = np.concatenate([[0], np.cumsum(qs)]).astype(np.int64)
    hs0 = inputs.normal_bf16(8, (int(cu[-1]), hidden))
    h = tdev(hs0)
    for l in range(layers):
        nxt = torch.empty_like(h)
        kvr.kvr_layer_forward(C.ctx, l, ld, devs[l][1], seqs, [L] * len(qs), cu, h, nxt, ws)
        h = nxt
    kvr.kvr_seq_advance(C.ctx, seqs, qs)
    got_suffix = bits_of(h)
    # ---- one decode token per consumer
    hd0 = inputs.normal_bf16(9, (len(qs), hidden))
    hd = tdev(hd0)
    for l in range(layers):
        nxt = torch.empty_like(hd)
        kvr.kvr_layer_forward(C.ctx, l, ld, devs[l][1], seqs, [L + q for q in qs], list(range(len(qs) + 1)),
                              hd, nxt, ws)
        hd = nxt
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK, kvr.kvr_last_error()
    got_dec = bits_of(hd)
    for b, q in enumerate(qs):
        hb, hdb = hs0[cu[b]:cu[b + 1]], hd0[b:b + 1]
        for l in range(layers):
            kb, vb = caches[l]
            hb, ks, vs, _ = oracle.layer_forward(hb, Ws[l], L + np.arange(q), kb, vb, Hq, Hkv, THETA, EPS)
            hdb, _, _, _ = oracle.layer_forward(hdb, Ws[l], [L + q], np.concatenate([kb, ks]),
                                                np.concatenate([vb, vs]), Hq, Hkv, THETA, EPS)
        check_layer(got_suffix[cu[b]:cu[b + 1]], hb, f"reuse step, consumer {b}", layers)
        check_layer(got_dec[b:b + 1], hdb, f"decode step, consumer {b}", layers)
    C.close()


def test_layer_small_two_layers(kvr):
    run_case(kvr, layers=2, hidden=256, inter=512, Hq=8, Hkv=2, d=64, L=300, qs=[37, 5])


def test_layer_qwen3_4b_shape(kvr):
    """Qwen3-4B layer widths (hidden 2560, MLP 9728, 32 / 8 heads x 128), the
    3774-token document, a 64-token continuation and a decode token."""
    run_case(kvr, layers=1, hidden=2560, inter=9728, Hq=32, Hkv=8, d=128, L=3774, qs=[64])
