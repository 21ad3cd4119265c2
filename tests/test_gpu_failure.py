"""Failure detection on the GPU without a GPU fault: a device-side wait that
runs out (a barrier phase nothing completes) is reported through the
context's error word as KVR_ERR_TIMEOUT, the word is cleared by the read, and
the context keeps working afterwards."""
import numpy as np
import pytest

from harness import bits_of, tdev
from paper_2606_13361_gb300 import inputs

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def kvr():
    from paper_2606_13361_gb300 import kvr as k
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return k


def test_device_wait_timeout_is_reported_and_the_context_survives(kvr):
    C = kvr.Context(kvr.make_desc(1, 4, 1, 64, max_positions=1024), n_pages=8, max_seqs=4)
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK
    kvr.kvr_selftest_wait_timeout(C.ctx)
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_ERR_TIMEOUT
    assert "time limit" in kvr.kvr_last_error()
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK  # the read cleared the word
    art = inputs.normal_bf16(2, (1, 2, 1, 10, 64))
    p = kvr.kvr_load_kv(C.ctx, kvr.kvr_artifact_meta(C.desc.model_id, 1, 10), tdev(art), True)
    out = torch.empty(art.nbytes, dtype=torch.uint8, device="cuda")
    kvr.kvr_export_kv(C.ctx, p, out, True)
    assert kvr.kvr_sync_status(C.ctx) == kvr.KVR_OK
    assert np.array_equal(bits_of(out.view(torch.bfloat16)).reshape(art.shape), art)
    C.close()
