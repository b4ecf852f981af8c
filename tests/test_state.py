"""Checkpoint and resume of the feedback state a decoding loop carries from
step to step (the trigger's entropy history, the selection's EMA score
table): host logic of ``VerifyStep`` on CPU buffers, no kernel launched."""
import numpy as np
import pytest

import synth


@pytest.fixture(scope="module")
def mods():
    from paper_2511_01282_gb300 import build
    build.build()
    from paper_2511_01282_gb300 import respec
    from paper_2511_01282_gb300.pipeline import VerifyStep, arrays_from_workload
    return respec, VerifyStep, arrays_from_workload


def _step(mods, seed, B):
    rs, VerifyStep, arrays_from_workload = mods
    w = synth.build(synth.small_spec(B=B, V=400), seed=seed)
    s = w.spec
    return VerifyStep(arrays_from_workload(w), rs.params(**s.params()), s.Hq, s.Hkv, s.D,
                      pos_cap=s.pos_cap, device="cpu")


def test_state_round_trip(mods, tmp_path):
    a = _step(mods, 1, 3)
    a.d["hist"].add_(0.25)
    a.d["hist_n"].fill_(2)
    a.d["scores"].mul_(0.5)
    snap = a.state()
    a.save_state(tmp_path / "state.npz")
    b = _step(mods, 1, 3)
    for k in b.STATE_KEYS:  # a fresh batch starts from its inputs
        assert (b.d[k].numpy() == b.host[k]).all()
    b.load_state_file(tmp_path / "state.npz")
    for k in b.STATE_KEYS:
        got = b.d[k].numpy()
        assert got.dtype == snap[k].dtype and (got == snap[k]).all(), k
    b.reset_state()
    for k in b.STATE_KEYS:
        assert (b.d[k].numpy() == b.host[k]).all()


def test_state_of_another_batch_shape_is_refused(mods):
    a = _step(mods, 1, 3)
    b = _step(mods, 2, 4)
    before = {k: v.copy() for k, v in b.state().items()}
    with pytest.raises(ValueError, match="hist"):
        b.load_state(a.state())
    for k in b.STATE_KEYS:  # nothing was written
        assert (b.d[k].numpy() == before[k]).all()
    bad = a.state()
    bad["scores"] = bad["scores"].astype(np.float64)
    with pytest.raises(ValueError, match="scores"):
        a.load_state(bad)
