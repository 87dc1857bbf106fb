"""The device GELU forms against the exact erf form (App. C.2: phi = GELU), on a
dense grid u in [-12, 12] (step 1e-3) at several gate values, through
mot_debug_gelu. The reference is the oracle's erf GELU in double; the bound
of each form is stated below with what sets it."""
import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

import _gpu as G   # noqa: E402
M = G.M

U = np.round(np.arange(-12000, 12001) * 1e-3, 12)
GATES = (1.0, 0.5, 0.13, 0.9)
_REF = None


def reference():
    """GELU(u) in double from the oracle (its erf form is pinned to the
    standard-normal table)."""
    global _REF
    if _REF is None:
        _REF = np.array([oracle.gelu(float(np.float32(x))) for x in U])
    return _REF


def run(form, g):
    u32 = U.astype(np.float32)
    u = torch.from_numpy(u32).cuda()
    gate = torch.full_like(u, g)
    out = torch.empty_like(u)
    M.mot_debug_gelu(form, u, gate, out)
    torch.cuda.synchronize()
    return out.cpu().numpy().astype(np.float64)


def ulp16(x):
    """Spacing of fp16 at |x| (the rounding step of the fp16 result)."""
    return np.spacing(np.abs(x).astype(np.float16)).astype(np.float64)


@pytest.mark.parametrize("g", GATES)
def test_tensor_core_mlp_gelu(g):
    """Form 0 rounds u to fp16 and evaluates the tanh form in packed fp16x2.
    Its error is the tanh form's (at most 4.7e-4 at |u| = 2.7), the fp16 tanh
    near -1 (1 + t loses the bits of t below 2^-11 for u < -1.5: up to about
    8e-4 at g = 1), and the fp16 rounding of u and of the result (one fp16
    step of the result for u > 1). Bound: 1.2e-3 * g + 2 fp16 steps of the
    result."""
    ref = reference() * g
    got = run(M.GELU_FORM_MLP, g)
    err = np.abs(got - ref)
    bound = 1.2e-3 * g + 2 * ulp16(ref)
    i = int(np.argmax(err - bound))
    neg = U < 0
    print(f"form 0 g={g}: max abs {err.max():.3e} at u={U[np.argmax(err)]}, "
          f"u<0 max abs {err[neg].max():.3e} at u={U[neg][np.argmax(err[neg])]}, "
          f"|u|<=1 max abs {err[np.abs(U) <= 1].max():.3e}")
    assert np.isfinite(got).all()
    assert (err <= bound).all(), f"u={U[i]}: got {got[i]}, want {ref[i]}, bound {bound[i]}"


@pytest.mark.parametrize("g", GATES)
def test_backbone_gelu(g):
    """Form 1: the tanh form in fp32 on the hardware tanh unit. Its error is the
    tanh form's 4.7e-4 plus the approximate tanh near -1. Bound: 1.2e-3 * g
    + 1e-3 of the result."""
    ref = reference() * g
    got = run(M.GELU_FORM_BACKBONE, g)
    err = np.abs(got - ref)
    bound = 1.2e-3 * g + 1e-3 * np.abs(ref)
    i = int(np.argmax(err - bound))
    print(f"form 1 g={g}: max abs {err.max():.3e} at u={U[np.argmax(err)]}")
    assert (err <= bound).all(), f"u={U[i]}: got {got[i]}, want {ref[i]}, bound {bound[i]}"


@pytest.mark.parametrize("g", GATES)
def test_simt_gelu_is_the_erf_form(g):
    """Form 2: erff in fp32 (SIMT path, fp32 workloads). Bound: 1e-6 of the
    result + 2e-7 * g."""
    ref = reference() * g
    got = run(M.GELU_FORM_SIMT, g)
    err = np.abs(got - ref)
    bound = 1e-6 * np.abs(ref) + 2e-7 * g
    i = int(np.argmax(err - bound))
    print(f"form 2 g={g}: max abs {err.max():.3e} at u={U[np.argmax(err)]}")
    assert (err <= bound).all(), f"u={U[i]}: got {got[i]}, want {ref[i]}, bound {bound[i]}"


def test_probe_rejects_bad_arguments():
    u = torch.zeros(4, device="cuda")
    with pytest.raises(M.MotError):
        M.mot_debug_gelu(3, u, u, u)
