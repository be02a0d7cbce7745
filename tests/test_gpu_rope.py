"""Compaction with K moved to receiver positions by the rotary embedding (GPU).

V must be copied byte for byte; K must match the oracle (rotation in double, one rounding to
bf16) to within one bf16 step, and exactly wherever the rotation angle is zero.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_32046_gb300 as cb
import synth
from gpu_helpers import make_cb

pytestmark = pytest.mark.gpu


def _run(shape, Ts, m):
    w = synth.custom_workload(synth.Shape(*shape), Ts, m, seed=17, n_planted_spans=2)
    c = make_cb(w.spec.shape, max(Ts), m, len(Ts))
    pairs = [(s.K.cuda(), s.V.cuda()) for s in w.senders]
    qs = [w.queries[s.task].cuda() for s in w.senders]
    f = cb.Filter(c, pairs, qs, 0.3).run()
    c.sync_status()
    return c, f


def _bits(t):
    return t.cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def _f32(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


@pytest.mark.parametrize("style", [0, 1])
@pytest.mark.parametrize("shape,pos0,base", [((2, 8, 2, 128), 500, 1e6), ((2, 8, 4, 64), 200000, 1e4)])
def test_rope_compaction_matches_oracle(shape, pos0, base, style):
    c, f = _run(shape, [300, 517, 64], 12)
    f.compact(rope=dict(base=base, style=style, pos0=pos0))
    c.sync_status()
    o = oracle.default()
    ko, vo = _bits(f.k_out), _bits(f.v_out)
    total = exact = 0
    for i in range(len(f.Ts)):
        B, off = f.budgets[i], f.offsets[i]
        idx = f.idx[i][:B].cpu().numpy()
        rk, rv = o.compact_rope(f.Ks[i].cpu(), f.Vs[i].cpu(), idx, base, style, pos0=pos0, offset=off)
        assert np.array_equal(vo[:, :, off:off + B], rv[:, :, off:])
        got, want = ko[:, :, off:off + B], rk[:, :, off:]
        # one bf16 step of the result (2^-7 relative), plus the absolute float error of a
        # rotation of O(1) inputs for results that nearly cancel
        err = np.abs(_f32(got) - _f32(want))
        assert np.all(err <= np.abs(_f32(want)) * 2.0 ** -7 + 1e-5), float(err.max())
        total += got.size
        exact += int((got == want).sum())
    assert exact >= 0.97 * total, exact / total


def test_zero_rotation_is_the_identity():
    c, f = _run((1, 8, 2, 128), [300], 12)
    K, V = f.Ks[0], f.Vs[0]
    idx = torch.arange(5, 45, dtype=torch.int32, device="cuda")
    ko = torch.zeros(1, 2, 40, 128, dtype=torch.bfloat16, device="cuda")
    vo = torch.zeros_like(ko)
    c.compact_rope([K], [V], [idx], [40], ko, vo, [0], base=1e6, style=0, pos0=5)   # position t -> t
    c.sync_status()
    assert torch.equal(ko.view(torch.int16), K[:, :, 5:45].view(torch.int16))
    assert torch.equal(vo.view(torch.int16), V[:, :, 5:45].view(torch.int16))


def test_bad_rope_arguments():
    c, f = _run((1, 8, 2, 128), [300], 12)
    for base, style in ((0.5, 0), (1e4, 2), (float("inf"), 0)):
        with pytest.raises(cb.CBError, match="CB_EINVAL"):
            f.compact(rope=dict(base=base, style=style, pos0=0))
