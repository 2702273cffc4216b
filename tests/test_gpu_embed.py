"""The embedding gather (vt_embed) through the C ABI: every row is the table row of its id, bit for
bit; ids outside [0, vocab) give a zero row and raise VT_DEV_BAD_TOKEN in the model's status word.
"""
from __future__ import annotations

import numpy as np
import pytest

import synthetic
from tests.parity import shapes_of

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _model(vt, wl):
    shapes = shapes_of(vt, wl)
    return vt.vt_model_create(shapes, None, wl.embedding())


@pytest.mark.parametrize("cid", [1, 5])
def test_embed_rows_are_table_rows_bit_for_bit(vtlib, cid):
    """Seeded ids (uniform over the vocabulary, as the prompt generator draws them) plus the ends
    of the range: 0 and vocab - 1.  Config 5 has the 128256-row Llama-3 vocabulary."""
    vt = vtlib
    wl = synthetic.WORKLOADS[cid]
    table = wl.embedding()
    ids = np.concatenate([wl.token_ids(509, stream=41), [0, wl.vocab - 1, 0]]).astype(np.int32)
    m = _model(vt, wl)
    try:
        out = torch.full((ids.size, wl.d_model), 7.0, dtype=torch.float16, device="cuda")
        vt.vt_embed(m, torch.from_numpy(ids).cuda(), out)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        assert np.array_equal(got.view(np.uint16), table[ids].view(np.uint16))
        assert vt.vt_model_status(m) == 0
    finally:
        vt.vt_model_destroy(m)


def test_embed_out_of_range_ids_give_zero_rows_and_set_the_status(vtlib):
    vt = vtlib
    wl = synthetic.WORKLOADS[1]
    table = wl.embedding()
    ids = np.array([5, -1, wl.vocab, 31999, np.iinfo(np.int32).min, np.iinfo(np.int32).max, 0],
                   dtype=np.int32)
    m = _model(vt, wl)
    try:
        out = torch.full((ids.size, wl.d_model), 3.0, dtype=torch.float16, device="cuda")
        vt.vt_embed(m, torch.from_numpy(ids).cuda(), out)
        torch.cuda.synchronize()
        got = out.cpu().numpy().view(np.uint16)
        valid = (ids >= 0) & (ids < wl.vocab)
        assert np.array_equal(got[valid], table[ids[valid]].view(np.uint16))
        assert not got[~valid].any(), "out-of-range ids must give +0.0 rows"
        assert vt.vt_model_status(m, clear=True) == vt.VT_DEV_BAD_TOKEN
        assert vt.vt_model_status(m) == 0
        # a clean gather leaves the word clear
        vt.vt_embed(m, torch.from_numpy(ids[valid]).cuda(), out[: int(valid.sum())])
        assert vt.vt_model_status(m) == 0
    finally:
        vt.vt_model_destroy(m)


def test_embed_argument_errors(vtlib):
    vt = vtlib
    wl = synthetic.WORKLOADS[1]
    shapes = shapes_of(vt, wl)
    m = vt.vt_model_create(shapes, None, None)  # the table is never loaded
    try:
        ids = torch.zeros(4, dtype=torch.int32, device="cuda")
        out = torch.empty((4, wl.d_model), dtype=torch.float16, device="cuda")
        with pytest.raises(vt.VtError) as e:
            vt.vt_embed(m, ids, out)
        assert e.value.status == vt.VT_ERR_STATE
        vt.vt_model_load_embedding(m, wl.embedding())
        vt.vt_embed(m, ids[:0], out[:0])  # n = 0 enqueues nothing
        torch.cuda.synchronize()
    finally:
        vt.vt_model_destroy(m)
