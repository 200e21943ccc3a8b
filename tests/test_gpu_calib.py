"""GPU parity of the SeqCalib candidate replay (hwkv_calib_scores) against the
oracle's Eq. conditional-similarity: every individual cosine and every
per-head mean score, and the threshold selection made from them."""
import numpy as np
import pytest

import hwkv_gen
import oracle
import paper_2609_02029_gb300 as hwkv

pytestmark = pytest.mark.gpu

COS_ATOL = 5e-3    # individual cos_eval of fp32 outputs (bf16 inputs, fp32 accumulation)
SCORE_ATOL = 2e-3  # means over (position, query head)


def _trace(g, N, T, Hkv, Hq, d, pos):
    """Device q [N][P][Hq][d] and head-major k, v [N][Hkv][T][d]; host copies for the oracle."""
    import torch
    s = torch.cuda.current_stream().cuda_stream
    K = torch.empty((N, T, Hkv, d), dtype=torch.bfloat16, device="cuda")
    V = torch.empty_like(K)
    hwkv_gen.fill_device(g, hwkv_gen.K, 0, N, 0, T, Hkv, d, K.data_ptr(), s)
    hwkv_gen.fill_device(g, hwkv_gen.V, 0, N, 0, T, Hkv, d, V.data_ptr(), s)
    Kh = K.permute(0, 2, 1, 3).contiguous()
    Vh = V.permute(0, 2, 1, 3).contiguous()
    P = pos.shape[1]
    Q = np.stack([np.stack([hwkv_gen.fill_host(g, hwkv_gen.Q, 0, N, int(pos[n, p]), 1, Hq, d)[n, 0]
                            for p in range(P)]) for n in range(N)])  # [N][P][Hq][d]
    Qd = torch.from_numpy(Q.view(np.int16)).view(torch.bfloat16).cuda()
    Khost = K.view(torch.int16).cpu().numpy().view(np.uint16)  # [N][T][Hkv][d]
    Vhost = V.view(torch.int16).cpu().numpy().view(np.uint16)
    return Qd, Kh, Vh, Q, Khost, Vhost


@pytest.mark.parametrize("N,P,T,Hkv,Hq,d,windows", [
    (2, 5, 3000, 2, 8, 64, [16, 200, 1000]),
    (1, 6, 2500, 2, 12, 256, [64, 512]),          # G = 6, d = 256
    (1, 4, 1800, 1, 8, 128, [1, 2, 4, 8, 16, 32, 64, 1500]),  # K = 8, G = 8
    (2, 3, 700, 3, 3, 128, [100]),                 # G = 1, K = 1
])
def test_calib_scores_match_oracle(N, P, T, Hkv, Hq, d, windows):
    import torch
    g = hwkv_gen.desc(17, per_head_scale=True)
    rng = np.random.default_rng(5)
    pos = np.sort(rng.integers(T // 2, T, size=(N, P)), axis=1)
    pos[0, 0] = 0 if T < 1000 else pos[0, 0]  # a position with a single key
    Qd, Kh, Vh, Q, Khost, Vhost = _trace(g, N, T, Hkv, Hq, d, pos)
    desc = hwkv.make_calib_desc(N, P, Hkv, Hq, d, T, windows, pos)
    nbytes = hwkv.hwkv_calib_workspace_bytes(desc)
    ws = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    scale = 1.0 / np.sqrt(d)
    scores, cos = hwkv.hwkv_calib_scores(desc, Qd, Kh, Vh, scale, ws, nbytes, with_cos=True)
    G = Hq // Hkv
    want_scores = np.zeros((Hkv, len(windows)))
    for h in range(Hkv):
        rows_q, rows_p, got_c = [], [], []
        for n in range(N):
            for p in range(P):
                for gg in range(G):
                    rows_q.append(Q[n, p, h * G + gg])
                    rows_p.append(pos[n, p])
                    got_c.append(cos[n, p, h * G + gg])
        # one oracle call per sequence (its K/V history), rows of that sequence
        acc = []
        for n in range(N):
            sl = slice(n * P * G, (n + 1) * P * G)
            s_n, c_n = oracle.conditional_similarity_bf16(
                np.stack(rows_q[sl]), rows_p[sl], Khost[n, :, h], Vhost[n, :, h], windows, scale)
            np.testing.assert_allclose(np.stack(got_c[sl]), c_n, atol=COS_ATOL, rtol=0)
            acc.append(c_n)
        want_scores[h] = np.concatenate(acc).mean(axis=0)
    np.testing.assert_allclose(scores, want_scores, atol=SCORE_ATOL, rtol=0)
    # selection: floors placed away from every score so both sides must agree
    flat = np.sort(np.unique(np.round(want_scores.ravel(), 6)))
    floors = [0.5] + [(a + b) / 2 for a, b in zip(flat[:-1], flat[1:]) if b - a > 4 * SCORE_ATOL]
    for tau in floors:
        got = hwkv.hwkv_calib_select(scores, windows, T, tau)
        want = [oracle.select_window(want_scores[h], windows, T, tau) for h in range(Hkv)]
        assert list(got) == want


def test_trace_check_accepts_matching_trace_and_rejects_wrong_mapping():
    # the traced full-history outputs (here: the oracle's full-window attention) must be
    # reproduced by the replay; a trace whose query heads read the wrong KV head (a GQA
    # mapping mismatch) must fail the 0.99 check (App. "Experimental Protocol")
    import torch
    N, P, T, Hkv, Hq, d = 2, 4, 1500, 2, 8, 128
    g = hwkv_gen.desc(23, per_head_scale=True)
    pos = np.sort(np.random.default_rng(3).integers(T // 2, T, size=(N, P)), axis=1)
    Qd, Kh, Vh, Q, Khost, Vhost = _trace(g, N, T, Hkv, Hq, d, pos)
    G = Hq // Hkv
    scale = 1.0 / np.sqrt(d)

    def traced_outputs(kv_of_q):
        out = np.zeros((N, P, Hq, d), dtype=np.float32)
        for n in range(N):
            for qh in range(Hq):
                h = kv_of_q(qh)
                O, _ = oracle.window_attention_bf16(Q[n, :, qh], pos[n], Khost[n, :, h],
                                                    Vhost[n, :, h], 0, scale)
                out[n, :, qh] = O
        return torch.from_numpy(out).cuda()

    desc = hwkv.make_calib_desc(N, P, Hkv, Hq, d, T, [64, 512], pos)
    nbytes = hwkv.hwkv_calib_workspace_bytes(desc)
    ws = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    m, per = hwkv.hwkv_calib_trace_check(desc, Qd, Kh, Vh, scale, traced_outputs(lambda q: q // G),
                                         ws, nbytes)
    assert m > 0.999 and per.min() == np.float32(m)
    with pytest.raises(hwkv.HwkvError) as e:
        hwkv.hwkv_calib_trace_check(desc, Qd, Kh, Vh, scale,
                                    traced_outputs(lambda q: (q // G + 1) % Hkv), ws, nbytes)
    assert e.value.status == hwkv.HWKV_ETRACE
