"""kvr_reuse_attn_noalloc: reuse attention for callers that cannot allocate
device memory where they run attention (code under another framework's
allocator that forbids side allocations, a runtime that reserved all device
memory up front).  Its split partials live in a fixed array inside the
library's device image instead of a caller-provided workspace.

Through the C ABI, on the GPU: the variant returns what kvr_reuse_attn returns
(within the tolerance the parity tests use) on two calls in a row -- the second
call finds the first call's partials still in the shared array -- and an
explicit split count whose partials do not fit the array is refused."""
import numpy as np
import pytest

from harness import check_close, f64_of, tdev
from paper_2606_13361_gb300 import inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

HQ, HKV, D = 32, 8, 128


def _consumers(kvr, C, L, qs, seed):
    """A loaded stand-in prefix of L positions, one fork per consumer, and the
    consumers' suffix tokens appended; returns (seqs, cu_q, q_out)."""
    art = inputs.normal_bf16(seed, (1, 2, HKV, L, D))
    p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, 1, L), tdev(art), True)
    seqs = [kvr.kvr_seq_fork(C.ctx, p) for _ in qs]
    li = inputs.layer_inputs(seed + 1, int(sum(qs)), HQ, HKV, D)
    cu = np.concatenate([[0], np.cumsum(qs)]).astype(np.int64)
    q_out = torch.empty((int(cu[-1]), HQ, D), dtype=torch.bfloat16, device="cuda")
    kvr.kvr_append_kv(C.ctx, 0, seqs, [L] * len(qs), cu, tdev(li.q_pre), tdev(li.k_pre), tdev(li.v),
                      tdev(li.q_norm_w), tdev(li.k_norm_w), q_out)
    return seqs, cu, q_out


def _both(kvr, C, seqs, cu, q, splits):
    ref = torch.empty_like(q)
    got = torch.empty_like(q)
    lref = torch.empty((q.shape[0], HQ), dtype=torch.float32, device="cuda")
    lgot = torch.empty_like(lref)
    kvr.kvr_reuse_attn(C.ctx, 0, seqs, cu, q, ref, lref, num_splits=splits)
    kvr.kvr_reuse_attn_noalloc(C.ctx, 0, seqs, cu, q, got, lgot, num_splits=splits)
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK, kvr.kvr_last_error()
    return ref, got, lref, lgot


def test_noalloc_matches_reuse_attn_on_two_calls_in_a_row():
    from paper_2606_13361_gb300 import kvr
    assert torch.cuda.is_available()
    C = kvr.Context(kvr.make_desc(1, HQ, HKV, D, max_positions=8192), n_pages=96, max_seqs=16)
    seqs, cu, q = _consumers(kvr, C, 1000, [1, 17, 64], seed=21)
    # call 1: a prefill-sized batch of three consumers, automatic splits
    ref, got, lref, lgot = _both(kvr, C, seqs, cu, q, splits=0)
    check_close(f64_of(got), f64_of(ref), "no-alloc call 1")
    np.testing.assert_allclose(lgot.cpu().numpy(), lref.cpu().numpy(), rtol=0, atol=1e-4)
    # call 2 right after: a different batch (one decode token each) and an
    # explicit split count, reusing the same scratch
    kvr.kvr_seq_advance(C.ctx, seqs, [1, 17, 64])
    li = inputs.layer_inputs(33, 3, HQ, HKV, D)
    q2 = torch.empty((3, HQ, D), dtype=torch.bfloat16, device="cuda")
    starts = [kvr.kvr_seq_length(C.ctx, s) for s in seqs]
    kvr.kvr_append_kv(C.ctx, 0, seqs, starts, [0, 1, 2, 3], tdev(li.q_pre), tdev(li.k_pre), tdev(li.v),
                      tdev(li.q_norm_w), tdev(li.k_norm_w), q2)
    ref2, got2, lref2, lgot2 = _both(kvr, C, seqs, [0, 1, 2, 3], q2, splits=5)
    check_close(f64_of(got2), f64_of(ref2), "no-alloc call 2")
    np.testing.assert_allclose(lgot2.cpu().numpy(), lref2.cpu().numpy(), rtol=0, atol=1e-4)
    C.close()


def test_noalloc_refuses_partials_larger_than_its_scratch():
    from paper_2606_13361_gb300 import kvr
    C = kvr.Context(kvr.make_desc(1, HQ, HKV, D, max_positions=8192), n_pages=96, max_seqs=16)
    seqs, cu, q = _consumers(kvr, C, 2000, [530], seed=41)
    # 2 splits x 530 rows x 32 heads x 129 x 4 B > 16 MiB
    per_split = 530 * HQ * (D + 1) * 4
    assert 2 * per_split > kvr.KVR_NOALLOC_SCRATCH_BYTES
    out = torch.empty_like(q)
    with pytest.raises(kvr.KvrError) as e:
        kvr.kvr_reuse_attn_noalloc(C.ctx, 0, seqs, cu, q, out, num_splits=2)
    assert e.value.status == kvr.KVR_ERR_OOM and "scratch" in str(e.value)
    # automatic splits stay within the scratch and match the regular call
    ref, got, _, _ = _both(kvr, C, seqs, cu, q, splits=0)
    check_close(f64_of(got), f64_of(ref), "no-alloc automatic splits")
    C.close()


def test_noalloc_empty_splits_never_read_an_earlier_calls_partials():
    """Every partial a call reads back, the same call wrote, including the
    partials of splits that have no keys: consecutive calls over 64 rows with
    6, 14 and 3 splits, where the later calls' partials (and their lse rows)
    lie over the earlier calls' leftovers, and where one query block (a fresh
    sequence of 32 tokens, one key tile) leaves most splits empty.  Each call
    equals kvr_reuse_attn with the same split count bit for bit."""
    from paper_2606_13361_gb300 import kvr
    from harness import bits_of
    C = kvr.Context(kvr.make_desc(1, HQ, HKV, D, max_positions=8192), n_pages=128, max_seqs=16)
    L = 4000
    art = inputs.normal_bf16(61, (1, 2, HKV, L, D))
    p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, 1, L), tdev(art), True)
    c1, c2, c3 = (kvr.kvr_seq_fork(C.ctx, p) for _ in range(3))
    x = kvr.kvr_seq_open(C.ctx)

    def append(seqs, starts, seed):
        li = inputs.layer_inputs(seed, 32 * len(seqs), HQ, HKV, D)
        q = torch.empty((32 * len(seqs), HQ, D), dtype=torch.bfloat16, device="cuda")
        kvr.kvr_append_kv(C.ctx, 0, seqs, starts, [32 * i for i in range(len(seqs) + 1)], tdev(li.q_pre),
                          tdev(li.k_pre), tdev(li.v), tdev(li.q_norm_w), tdev(li.k_norm_w), q)
        return q

    qa = append([c1, c2], [L, L], 62)     # two consumers of the loaded prefix
    qb = append([c3, x], [L, 0], 63)      # one consumer, and a fresh sequence of 32 tokens
    cu = [0, 32, 64]
    for seqs, q, splits in (([c1, c2], qa, 6), ([c3, x], qb, 14), ([c3, x], qb, 3)):
        # 64 rows x 32 heads x 129 floats per split: 6, 14 and 3 splits fit the scratch
        assert splits * 64 * HQ * (D + 1) * 4 <= kvr.KVR_NOALLOC_SCRATCH_BYTES
        ref, got, lref, lgot = _both(kvr, C, seqs, cu, q, splits)
        assert np.array_equal(bits_of(got), bits_of(ref)), f"{splits} splits: outputs differ"
        assert np.array_equal(lgot.cpu().numpy().view(np.uint32), lref.cpu().numpy().view(np.uint32)), \
            f"{splits} splits: lse differs"
        assert np.isfinite(f64_of(got)).all()
    C.close()
