"""Resume from a checkpoint on the GPU: a run that is saved after some
optimisation steps and resumed in fresh buffers continues bit for bit like
the run that was never interrupted.

The checkpoint holds Theta_IF, the codes and the step counter only; W^ is
rebuilt on load by R_B and D_R with no mapping.  The quantizer kernels are
deterministic (fixed reduction orders, no atomics), so the comparison is
exact: parameters and W^ by bit pattern, codes by value.  The gradient
scale makes every remap step move codes (checked), so the resumed run
really depends on the stored codes.
"""

import numpy as np
import pytest
import torch

from paper_2506_03781_gb300 import api, checkpoint, synth
from paper_2506_03781_gb300.recon import NAMES, BlockReconstructor

pytestmark = pytest.mark.gpu
STEPS = 6


def _bits(t):
    return t.detach().cpu().contiguous().view(torch.int32) if t.dtype == torch.float32 else t.detach().cpu()


def _same(a, b):
    return torch.equal(_bits(a), _bits(b))


def _matrix(out, n_in, q, g, seed):
    rng = np.random.default_rng(seed)
    raw, _ = synth.bf16_round((rng.standard_t(4, (out, n_in)) * 0.014).astype(np.float32))
    d = torch.device("cuda", 0)
    Wd = api.weights_tensor(raw, d)
    P = api.empty_params(out, n_in, q, g, d)
    codes = torch.empty(out, n_in, dtype=torch.uint8, device=d)
    api.uq_init_params(Wd, q, g, P, codes, G=4, T=3)
    Gs = [torch.from_numpy((rng.standard_normal((out, n_in)) * 3e-3).astype(np.float32)).to(d)
          for _ in range(STEPS)]
    return Wd, P, codes, Gs


def _quantizer(Wd, q, g, P, codes):
    out, n_in = Wd.shape
    what = torch.full((out, n_in), float("nan"), device=Wd.device)
    G = torch.zeros(out, n_in, device=Wd.device)
    return api.Quantizer(Wd, q, g, P, codes, what, G), G, what


def _steps(qz, G, Gs, t0, t1, p, mode):
    for t in range(t0, t1):
        G.copy_(Gs[t])
        qz.train_step(t, p_period=p, map_mode=mode)


@pytest.mark.parametrize("out,n_in,q,g,mode", [
    (256, 1024, 3, 128, api.MAP_LOCAL_PERIODIC),
    (96, 2048, 2, 64, api.MAP_LOCAL_PERIODIC),
    (64, 512, 4, 32, api.MAP_FULL),
])
@pytest.mark.parametrize("t_save", [3, 4])
def test_resumed_steps_match_the_uninterrupted_run(tmp_path, out, n_in, q, g, mode, t_save):
    p = 2
    Wd, P0, codes0, Gs = _matrix(out, n_in, q, g, 11)
    # the uninterrupted run
    Pa = {k: v.clone() for k, v in P0.items()}
    ca = codes0.clone()
    qa, Ga, wa = _quantizer(Wd, q, g, Pa, ca)
    qa.fwd(0, p, mode)
    first = ca.clone()
    _steps(qa, Ga, Gs, 0, STEPS, p, mode)
    assert (ca != first).any(), "the steps moved no code: the test would not exercise the stored codes"
    # the same run, saved after t_save steps ...
    Pb = {k: v.clone() for k, v in P0.items()}
    cb = codes0.clone()
    qb, Gb, wb = _quantizer(Wd, q, g, Pb, cb)
    qb.fwd(0, p, mode)
    _steps(qb, Gb, Gs, 0, t_save, p, mode)
    path = tmp_path / "q.pt"
    checkpoint.save_state(path, {"w": (Pb, cb)}, t_save, q=q, g=g, p=p, map_mode=mode)
    # ... and resumed in fresh buffers that hold other values
    mats, step, meta = checkpoint.load_state(path)
    assert step == t_save and meta["q"] == q and meta["g"] == g
    Pc = {k: torch.full_like(v, 7.0) for k, v in P0.items()}
    cc = torch.full_like(codes0, 255)
    qc, Gc, wc = _quantizer(Wd, q, g, Pc, cc)
    checkpoint.restore_into(mats["w"], Pc, cc)
    checkpoint.rebuild_what(qc)
    torch.cuda.synchronize()
    assert _same(wc, wb), "W^ rebuilt without mapping differs from the saved run's W^"
    _steps(qc, Gc, Gs, step, STEPS, p, mode)
    torch.cuda.synchronize()
    for k in api.PARAM_NAMES:
        assert _same(Pc[k], Pa[k]), k
    assert torch.equal(cc, ca)
    assert _same(wc, wa)


@pytest.fixture
def no_tf32():
    old = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    yield
    torch.backends.cuda.matmul.allow_tf32 = old


def test_block_reconstructor_save_and_load(tmp_path, no_tf32):
    """Algorithm 1 on a tiny block: the state loaded into a fresh
    reconstructor equals the saved one bit for bit (W^ included) and carries
    the step counter; the next steps then follow the uninterrupted run (the
    block's own forward and backward run in torch, fp32)."""
    shape = synth.BLOCKS["tiny"]
    q, g = 3, 32
    Wb = synth.block_weights(shape, 0)
    stored = {n: Wb[n][0] for n in NAMES}
    d = torch.device("cuda", 0)
    X, Xh = synth.block_inputs(shape, 2, 0, perturb=0.02)
    Xd = [torch.from_numpy(x).to(d) for x in X]
    Xhd = [torch.from_numpy(x).to(d) for x in Xh]

    ra = BlockReconstructor(shape, stored, q, g, device=d, compute_dtype=torch.float32, G=4, T=3)
    Yd = ra.targets(Xd)
    la = [float(ra.step(Yd[t % 2], Xhd[t % 2])) for t in range(4)]

    rb = BlockReconstructor(shape, stored, q, g, device=d, compute_dtype=torch.float32, G=4, T=3)
    lb = [float(rb.step(Yd[t % 2], Xhd[t % 2])) for t in range(2)]
    path = tmp_path / "block.pt"
    rb.save(path)

    rc = BlockReconstructor(shape, stored, q, g, device=d, compute_dtype=torch.float32, init=False)
    rc.load(path)
    assert rc.t == 2
    Pb, Cb, Wb_hat = rb.state()
    Pc, Cc, Wc_hat = rc.state()
    for n in NAMES:
        for k in api.PARAM_NAMES:
            assert np.array_equal(Pc[n][k].view(np.uint32), Pb[n][k].view(np.uint32)), (n, k)
        assert np.array_equal(Cc[n], Cb[n]), n
        assert np.array_equal(Wc_hat[n].view(np.uint32), Wb_hat[n].view(np.uint32)), n
    lc = [float(rc.step(Yd[t % 2], Xhd[t % 2])) for t in range(2, 4)]
    # torch's attention backward may sum in a run-dependent order, so the
    # runs agree to rounding from step 1 on
    assert lb[0] == la[0]
    for a, c in zip(la[1:], lb[1:] + lc):
        assert abs(a - c) <= 1e-6 * abs(a), (la, lb + lc)
    Pa, Ca, _ = ra.state()
    Pc, Cc, _ = rc.state()
    agree = np.mean(np.concatenate([(Cc[n] == Ca[n]).ravel() for n in NAMES]))
    assert agree >= 0.9999, agree
    for n in NAMES:
        for k in api.PARAM_NAMES:
            a, c = Pa[n][k].astype(np.float64), Pc[n][k].astype(np.float64)
            assert np.abs(a - c).max() <= 1e-6 * np.abs(a).max(), (n, k)


def test_load_rejects_another_bit_width(tmp_path):
    shape = synth.BLOCKS["tiny"]
    Wb = synth.block_weights(shape, 0)
    stored = {n: Wb[n][0] for n in NAMES}
    d = torch.device("cuda", 0)
    r3 = BlockReconstructor(shape, stored, 3, 32, device=d, compute_dtype=torch.float32, G=2, T=1)
    path = tmp_path / "b.pt"
    r3.save(path)
    r2 = BlockReconstructor(shape, stored, 2, 32, device=d, compute_dtype=torch.float32, init=False)
    with pytest.raises(ValueError):
        r2.load(path)
