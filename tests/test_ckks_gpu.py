"""End to end on the GPU, checked against float64 arithmetic only (the
paper's own check, Sec. 6 RQ1 "Exact Compilation": the compiled layer against
an FP64 computation): real slot vectors are encoded on the GPU
(fiona_encode), encrypted with a secret key on the host, the hybrid layer is
evaluated on the GPU (fiona_linear_eval, then fiona_linear_eval_rescale with
either quotient), and the decrypted, decoded outputs must equal the float64
slot-wise mat-vec within the CKKS error.  N = 2^10, three 40-bit primes,
Delta = 2^40; after the rescale the scale is Delta^2 / q_last."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

import oracle  # noqa: E402
from oracle import ckks_tiny  # noqa: E402
from paper_2609_35352_gb300 import build as B  # noqa: E402
from paper_2609_35352_gb300 import fiona as F  # noqa: E402
from paper_2609_35352_gb300 import workloads as W  # noqa: E402

from gpu_util import to_host  # noqa: E402

DELTA = 2.0 ** 40


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.build()
    oracle.build()


def mulmod(a, b, q):
    return (a.astype(object) * b.astype(object)) % q


def encode_gpu(ctx, L, vectors, scale):
    """Real slot vectors [count][N/2] -> NTT-form plaintexts [count][L][N] (fiona_encode)."""
    count, n = vectors.shape
    N = 2 * n
    slots = np.zeros((count, n, 2))
    slots[:, :, 0] = vectors
    c = torch.empty(count * N, dtype=torch.int64, device="cuda")
    w = torch.empty(count * N, dtype=torch.float64, device="cuda")
    out = torch.empty(count * L * N, dtype=torch.int64, device="cuda")
    ctx.encode(L, count, torch.from_numpy(slots).cuda(), scale, c, w, out)
    assert ctx.device_check() == F.FIONA_OK
    return to_host(out).reshape(count, L, N)


def ntt_of_ints(ctx, L, coeffs):
    """Integer polys [count][N] -> NTT form (fiona_encode_coeffs)."""
    count, N = coeffs.shape
    out = torch.empty(count * L * N, dtype=torch.int64, device="cuda")
    ctx.encode_coeffs(L, count, torch.from_numpy(np.ascontiguousarray(coeffs, dtype=np.int64)).cuda(), out)
    torch.cuda.synchronize()
    return to_host(out).reshape(count, L, N)


def decrypt_decode(ct, s_ntt, qs, scale):
    """ct [2][L'][N] (NTT form), s_ntt [L][N]: slots of c0 + c1 s, / scale."""
    Lp, N = ct.shape[1], ct.shape[2]
    coef = []
    for l in range(Lp):
        q = qs[l]
        d = (ct[0, l].astype(object) + mulmod(ct[1, l], s_ntt[l], q)) % q
        coef.append([int(v) for v in oracle.intt(np.array(d, dtype=np.uint64), q)])
    Q = 1
    for q in qs[:Lp]:
        Q *= q
    m = np.zeros(N)
    for k in range(N):
        Y = 0
        for l in range(Lp):
            Ml = Q // qs[l]
            Y = (Y + coef[l][k] * Ml * pow(Ml, -1, qs[l])) % Q
        m[k] = float(Y - Q if Y > Q // 2 else Y)
    e = np.array([pow(5, j, 2 * N) for j in range(N // 2)])
    vals = np.fft.ifft(np.concatenate([m, np.zeros(N)])) * (2 * N)
    return vals[e].real / scale


@pytest.mark.parametrize("round_", [False, True])
def test_encrypted_layer_matches_float64(round_):
    wl = W.make_workload("tiny", N=1024)
    plan_desc = wl.plan
    N, qs, L = wl.N, wl.moduli, wl.L
    n = N // 2
    rng = np.random.default_rng(2609)
    x = rng.uniform(-1, 1, (plan_desc.n_in, n))
    w = rng.uniform(-1, 1, (plan_desc.n_pt, n))
    for g in plan_desc.group_scale_pt:
        w[int(g)] = rng.uniform(0.05, 1.0, n)  # reconstruction factors are positive
    ctx = F.Context(N, qs, device=0)
    plan = F.Plan(ctx, plan_desc)

    # keys and ciphertexts: c1 = a, c0 = -a s + m + e (NTT form)
    s = rng.integers(-1, 2, (1, N))
    s_ntt = ntt_of_ints(ctx, L, s)[0]
    m = encode_gpu(ctx, L, x, DELTA)
    e = np.rint(rng.normal(0.0, 3.2, (plan_desc.n_in, N))).astype(np.int64)
    e_ntt = ntt_of_ints(ctx, L, e)
    cts = np.zeros((plan_desc.n_in, 2, L, N), np.uint64)
    for i in range(plan_desc.n_in):
        for l, q in enumerate(qs):
            a = rng.integers(0, q, N, dtype=np.uint64)
            c0 = (m[i, l].astype(object) + e_ntt[i, l].astype(object) - mulmod(a, s_ntt[l], q)) % q
            cts[i, 0, l] = np.array(c0, dtype=np.uint64)
            cts[i, 1, l] = a
    pts = encode_gpu(ctx, L, w, DELTA)

    d_in = torch.from_numpy(cts.view(np.int64)).cuda()
    d_pt = torch.from_numpy(pts.view(np.int64)).cuda()
    ref = ckks_tiny.float_layer(plan_desc, x, w)

    out = torch.empty(plan_desc.n_out * 2 * L * N, dtype=torch.int64, device="cuda")
    plan.eval(d_in, d_pt, out)
    work = torch.empty_like(out)
    res = torch.empty(plan_desc.n_out * 2 * (L - 1) * N, dtype=torch.int64, device="cuda")
    plan.eval_rescale(L, d_in, d_pt, work, res, round=round_)
    torch.cuda.synchronize()
    y = to_host(out).reshape(plan_desc.n_out, 2, L, N)
    yr = to_host(res).reshape(plan_desc.n_out, 2, L - 1, N)
    for j in range(plan_desc.n_out):
        err = np.max(np.abs(decrypt_decode(y[j], s_ntt, qs, DELTA ** 2) - ref[j]))
        assert err <= 1e-3, (j, err)
        err_r = np.max(np.abs(decrypt_decode(yr[j], s_ntt, qs, DELTA ** 2 / qs[-1]) - ref[j]))
        assert err_r <= 1e-3, (j, err_r)
