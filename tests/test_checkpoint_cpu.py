"""Checkpoint files of the quantizer state on the host (no GPU): Theta_IF,
the codes and the step counter round-trip bit for bit, and a file that does
not fit the buffers it is loaded into is rejected before anything is copied."""

import numpy as np
import pytest
import torch

from paper_2506_03781_gb300 import api, checkpoint


def _state(out, n_in, q, g, seed):
    gen = torch.Generator().manual_seed(seed)
    p = api.empty_params(out, n_in, q, g, device="cpu")
    for k in p:
        p[k].copy_(torch.randn(p[k].shape, generator=gen))
    codes = torch.randint(0, 1 << q, (out, n_in), generator=gen, dtype=torch.uint8)
    return p, codes


def test_round_trip_is_bit_exact(tmp_path):
    a = _state(8, 256, 3, 128, 0)
    b = _state(4, 512, 2, 64, 1)
    path = tmp_path / "state.pt"
    checkpoint.save_state(path, {"a": a, "b": b}, 7, q=3, g=128, p=2, lr_F=0.005, name="x")
    mats, step, meta = checkpoint.load_state(path)
    assert step == 7 and meta == {"q": 3, "g": 128, "p": 2, "lr_F": 0.005, "name": "x"}
    assert set(mats) == {"a", "b"}
    for name, (p, c) in (("a", a), ("b", b)):
        q = 3 if name == "a" else 2
        g = 128 if name == "a" else 64
        p2 = api.empty_params(*c.shape, q, g, device="cpu")
        c2 = torch.empty_like(c)
        checkpoint.restore_into(mats[name], p2, c2)
        for k in api.PARAM_NAMES:
            # bit patterns, so that a NaN or a signed zero would count too
            assert np.array_equal(p2[k].numpy().view(np.uint32), p[k].numpy().view(np.uint32)), (name, k)
        assert torch.equal(c2, c)


def test_snapshot_is_a_copy():
    p, c = _state(2, 128, 1, 128, 2)
    sp, sc = checkpoint.snapshot(p, c)
    p["delta"].fill_(0.0)
    c.fill_(0)
    assert not torch.equal(sp["delta"], p["delta"]) and sc.any()


@pytest.mark.parametrize("field", ["delta", "alpha", "s", "codes"])
def test_mismatched_buffers_are_rejected_untouched(tmp_path, field):
    src = _state(8, 256, 3, 128, 3)
    path = tmp_path / "s.pt"
    checkpoint.save_state(path, {"m": src}, 1)
    mats, _, _ = checkpoint.load_state(path)
    q = 2 if field == "alpha" else 3
    out = 4 if field in ("delta", "s", "codes") else 8
    p, c = _state(out, 256, q, 128, 4)
    before = {k: v.clone() for k, v in p.items()}, c.clone()
    with pytest.raises(ValueError):
        checkpoint.restore_into(mats["m"], p, c)
    assert all(torch.equal(p[k], before[0][k]) for k in p) and torch.equal(c, before[1])


def test_dtype_mismatch_is_rejected(tmp_path):
    src = _state(4, 128, 2, 128, 5)
    path = tmp_path / "s.pt"
    checkpoint.save_state(path, {"m": src}, 0)
    mats, _, _ = checkpoint.load_state(path)
    p, c = _state(4, 128, 2, 128, 6)
    with pytest.raises(ValueError):
        checkpoint.restore_into(mats["m"], p, c.to(torch.int32))


def test_other_files_and_bad_arguments_are_rejected(tmp_path):
    other = tmp_path / "other.pt"
    torch.save({"format": "something else"}, other)
    with pytest.raises(ValueError):
        checkpoint.load_state(other)
    st = _state(2, 128, 1, 128, 7)
    with pytest.raises(ValueError):
        checkpoint.save_state(tmp_path / "n.pt", {"m": st}, -1)
    with pytest.raises(TypeError):
        checkpoint.save_state(tmp_path / "m.pt", {"m": st}, 0, shape=[2, 128])
    p, c = st
    with pytest.raises(ValueError):
        checkpoint.save_state(tmp_path / "p.pt", {"m": ({k: v for k, v in p.items() if k != "zb"}, c)}, 0)
