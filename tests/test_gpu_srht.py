"""GPU parity of the EOGP-R second stage (the SRHT of App. B.2,
Eq. app_srht_definition) against the oracle.

* eogp_srht on fp32 rows: x within 1e-5 per-row relative error of the
  oracle's explicit Hadamard product, sign codes bit-exact outside the
  1e-4 ||x|| band, scales within 1e-5; padded widths (m not a power of two),
  k = 1 and k = p, a single row and many rows.
* The compression chain with the SRHT in place of P: the fp32 path (tiny
  layer) within 1e-5 and a GPT-2-shaped bf16 layer within 2e-3, codes and
  scales as for the PCA path.
* An out-of-range kept row is reported through the device status word.
"""
import numpy as np
import pytest

from oracle import eogp_oracle as O

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2609_37842_gb300 import eogp as E  # noqa: E402
from paper_2609_37842_gb300 import synth  # noqa: E402

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_37842_gb300 import build
    build.build()
    E.lib()
    yield
    torch.cuda.empty_cache()


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def row_rel(got, want):
    return np.linalg.norm(got - want, axis=1) / np.maximum(np.linalg.norm(want, axis=1), 1e-300)


def check_codes(x_or, codes, scales, k, tol):
    bits, sc = O.onebit(x_or)
    got = O.unpack_bits(codes.cpu().numpy().view(np.uint32), k)
    small = np.abs(x_or) < 1e-4 * np.linalg.norm(x_or, axis=1, keepdims=True)
    assert not ((got != bits) & ~small).any()
    np.testing.assert_allclose(scales.cpu().numpy(), sc, rtol=tol)


@pytest.mark.parametrize("B,m,k", [(3, 4096, 1024), (257, 1000, 1000), (1, 1, 1), (8, 8192, 8192),
                                   (5, 3000, 37)])
def test_srht_standalone(B, m, k):
    rng = np.random.default_rng(B * 31 + m)
    z = rng.standard_normal((B, m)).astype(np.float32)
    signs, rows = synth.srht_draw(m, k, seed=m + k)
    x = E.srht(dev(z), dev(signs), dev(rows))
    codes, scales = E.srht(dev(z), dev(signs), dev(rows), want_x=False, want_codes=True)
    E.sync_status()
    x_or = O.srht(z, signs, rows)
    rel = row_rel(x.cpu().numpy().astype(np.float64), x_or)
    print(f"max row rel err {rel.max():.2e}")
    assert rel.max() <= 1e-5
    check_codes(x_or, codes, scales, k, 1e-5)


def test_srht_out_of_range_row_sets_device_status():
    z = dev(np.ones((2, 100), np.float32))
    signs = dev(np.ones(100, np.int8))
    rows = dev(np.array([0, 5, 128], np.int32))        # p = 128: row 128 is out of range
    E.srht(z, signs, rows)
    with pytest.raises(E.EOGPError) as ei:
        E.sync_status()
    assert ei.value.code == E.EDEVICE
    E.sync_status()  # cleared


def srht_layer_check(w_dtype, d_in, d_out, T, B, m, k, tol, seed):
    rng = np.random.default_rng(seed)
    rnd = (lambda v: synth.round_to(v, w_dtype))
    tdt = torch.bfloat16 if w_dtype == "bf16" else torch.float32
    QA, QS = rnd(synth.haar_orthogonal(d_in, rng)), rnd(synth.haar_orthogonal(d_out, rng))
    lamA, lamS = synth.power_spectrum(d_in, 1.2), synth.power_spectrum(d_out, 1.2)
    a = rnd(rng.standard_normal((B, T, d_in)))
    s = rnd(rng.standard_normal((B, T, d_out)) * 0.1)
    signs, rows = synth.srht_draw(m, k, seed=seed)
    plan = E.Plan.from_factors(lamS, lamA, m, 0.1)
    VA = plan.gather_rows(0, dev(QA.T.astype(np.float32)).to(tdt))
    VS = plan.gather_rows(1, dev(QS.T.astype(np.float32)).to(tdt))
    sd, rd = dev(signs), dev(rows)
    desc = E.layer_desc(plan, T, k, VA, VS, None, srht_signs=sd, srht_rows=rd)
    ad, sdv = dev(a.astype(np.float32)).to(tdt), dev(s.astype(np.float32)).to(tdt)
    x = E.compress_layer(desc, ad, sdv, E.OUT_COORDS)
    codes, scales = E.compress_layer(desc, ad, sdv, E.OUT_CODES)
    E.sync_status()
    Lam = O.kfac_eigenvalues(lamS, lamA)
    z_or = O.first_stage(a, s, QA, QS, Lam, O.damping(Lam, 0.1), m)
    x_or = O.srht(z_or, signs, rows)
    rel = row_rel(x.cpu().numpy().astype(np.float64), x_or)
    print(f"max row rel err {rel.max():.2e}")
    assert rel.max() <= tol
    check_codes(x_or, codes, scales, k, max(tol, 1e-5))


def test_compress_srht_f32():
    srht_layer_check("f32", 64, 64, 16, 6, 512, 256, 1e-5, 3)


@pytest.mark.parametrize("k", [1024, 4096])
def test_compress_srht_bf16_gpt2_shape(k):
    srht_layer_check("bf16", 768, 768, 128, 3, 4096, k, 2e-3, 5 + k)
