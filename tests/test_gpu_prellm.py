"""Pre-LLM frame alignment on the GPU (Sec. 3.1, Eq. cka, Eq. gate) against
the literal fp64 oracle.

Tolerance: the kernels pool and accumulate the window Grams in fp32 over up
to 3584 features (relative rounding below 1e-5 for these inputs) and c_f is a
ratio of such sums; |c_gpu - c_oracle| <= 2e-4 covers it, and the same bound
applies to s_f and the normalised distance (affine in c_f and d_f)."""

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu
TOL = 2e-4


@pytest.fixture(scope="module")
def ap():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_08794_gb300 as ap
    return ap


def run(ap, vis, aud, F, tpf, dim, window, tau, beta):
    v_d = torch.from_numpy(vis.view(np.int16)).cuda()
    a_d = torch.from_numpy(aud.view(np.int16)).cuda()
    n = ap.apack_frame_alignment_workspace_size(F, dim)
    ws = torch.full((n + 256,), 0xA5, dtype=torch.uint8, device="cuda")   # no zeroed workspace needed
    off = (-ws.data_ptr()) % 256
    ws = ws[off:off + n]
    c = torch.empty(F, dtype=torch.float32, device="cuda")
    s = torch.empty_like(c)
    dn = torch.empty_like(c)
    cb = torch.empty(1, dtype=torch.float32, device="cuda")
    ap.apack_frame_alignment(v_d, a_d, F, tpf, aud.shape[0], dim, c, s, ws, window=window, tau=tau, beta=beta,
                             dnorm_out=dn, cbar_out=cb)
    torch.cuda.synchronize()
    return c.cpu().numpy(), s.cpu().numpy(), dn.cpu().numpy(), float(cb.item())


def inputs(seed, F, tpf, n_audio, dim):
    from synth.gen import normal_bf16_bits, TID_VIS_EMB, TID_AUD_EMB
    vis = normal_bf16_bits(seed, TID_VIS_EMB, 0, F * tpf * dim).reshape(F * tpf, dim)
    aud = normal_bf16_bits(seed, TID_AUD_EMB, 0, n_audio * dim).reshape(n_audio, dim)
    return vis, aud


CASES = [
    # F, tokens per frame, audio tokens, dim, window
    (1, 4, 3, 64, 3),
    (2, 3, 5, 8, 3),
    (5, 7, 63, 72, 5),
    (37, 16, 462, 256, 3),
    (20, 100, 250, 3584, 7),
    (9, 2, 9, 128, 1),
    (6, 3, 6, 4104, 3),       # rows wider than one CTA: separate pooling and CKA launches
]


@pytest.mark.parametrize("F,tpf,na,dim,window", CASES)
@pytest.mark.parametrize("tau", [0.0, 0.999])      # CKA branch, blend branch
def test_frame_alignment_matches_oracle(ap, F, tpf, na, dim, window, tau):
    vis, aud = inputs(F * 7 + dim, F, tpf, na, dim)
    c, s, dn, cb = run(ap, vis, aud, F, tpf, dim, window, tau, 0.9)
    ref = oracle.frame_alignment(vis, aud, F, tpf, window=window, tau=tau, beta=0.9)
    np.testing.assert_allclose(c, ref["c"], atol=TOL, rtol=0)
    np.testing.assert_allclose(dn, ref["dnorm"], atol=TOL, rtol=0)
    np.testing.assert_allclose(s, ref["s"], atol=TOL, rtol=0)
    assert cb == pytest.approx(ref["cbar"], abs=TOL)
    again = run(ap, vis, aud, F, tpf, dim, window, tau, 0.9)
    assert c.tobytes() == again[0].tobytes() and s.tobytes() == again[1].tobytes()


def test_frame_alignment_two_and_a_half_minute_clip(ap):
    # 300 frames of 100 visual tokens, 25 audio tokens per second at 2 fps, 7B hidden size
    F, tpf, na, dim = 300, 100, 3750, 3584
    vis, aud = inputs(11, F, tpf, na, dim)
    c, s, dn, cb = run(ap, vis, aud, F, tpf, dim, 3, 0.78, 0.9)
    ref = oracle.frame_alignment(vis, aud, F, tpf, window=3, tau=0.78, beta=0.9)
    np.testing.assert_allclose(c, ref["c"], atol=TOL, rtol=0)
    np.testing.assert_allclose(s, ref["s"], atol=TOL, rtol=0)


def test_frame_alignment_rejects_bad_arguments(ap):
    vis, aud = inputs(1, 4, 2, 8, 16)
    with pytest.raises(ap.ApackError):
        run(ap, vis, aud, 4, 2, 16, 4, 0.78, 0.9)        # even window
    with pytest.raises(ap.ApackError):
        run(ap, vis, aud[:3], 4, 2, 16, 3, 0.78, 0.9)    # fewer audio tokens than frames
