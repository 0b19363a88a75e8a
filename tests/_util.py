"""Shared test helpers: tolerance checks and chain conversion.  No arithmetic of
the method lives here (the oracle computes expected values, the library the
results under test)."""
import numpy as np
import torch

# Tolerances stated for this path: bf16 outputs |y - ref| <= 1e-2 + 1e-2 |ref|;
# fp32 outputs 1e-4 relative, read as |y - ref| <= 1e-4 |ref| + 1e-4 rms(ref)
# (a pure relative bound is undefined where ref crosses zero, e.g. after ReLU).
BF16_ATOL, BF16_RTOL = 1e-2, 1e-2
F32_RTOL = 1e-4


def to_np(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().double().numpy()


def check_bf16(got, ref, what=""):
    """bf16 outputs: the stated bound |y - ref| <= 1e-2 + 1e-2 |ref|, and the
    same bound with its absolute term scaled to the output, |y - ref| <=
    1e-2 (rms(ref) + |ref|).  The second is the one that bites when outputs are
    small (the N(0,1)/sqrt(K) workloads have rms ~ 0.02, where an absolute 1e-2
    would allow ~50% relative error).  Rounding an exact result to bf16 alone
    gives at most 2^-8 |ref|, well inside it.  A gate on max|y - ref| / rms(ref)
    alone is not used: over millions of outputs the largest |ref| reach ~5 rms
    and bf16 rounding by itself already takes that ratio to ~0.015."""
    got = to_np(got) if isinstance(got, torch.Tensor) else np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64).reshape(got.shape)
    err = np.abs(got - ref)
    bad = err > BF16_ATOL + BF16_RTOL * np.abs(ref)
    rms = float(np.sqrt(np.mean(ref ** 2))) if ref.size else 0.0
    assert not bad.any(), (f"{what}: {int(bad.sum())}/{bad.size} outside bf16 tolerance; "
                           f"max err {err.max():.3e} at {np.unravel_index(err.argmax(), err.shape)}")
    bad = err > BF16_RTOL * (rms + np.abs(ref))
    assert not bad.any(), (f"{what}: {int(bad.sum())}/{bad.size} outside 1e-2 (rms(ref) + |ref|), rms {rms:.3e}; "
                           f"max err {err.max():.3e} at {np.unravel_index(err.argmax(), err.shape)}")
    return float(err.max()) / max(rms, 1e-30) if ref.size else 0.0


def check_f32(got, ref, what=""):
    got = to_np(got) if isinstance(got, torch.Tensor) else np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64).reshape(got.shape)
    rms = float(np.sqrt(np.mean(ref ** 2))) if ref.size else 0.0
    err = np.abs(got - ref)
    bad = err > F32_RTOL * np.abs(ref) + F32_RTOL * rms
    assert not bad.any(), (f"{what}: {int(bad.sum())}/{bad.size} outside fp32 tolerance; "
                           f"max err {err.max():.3e}")
    return float(err.max()) / max(rms, 1e-30) if ref.size else 0.0


def chain_to(chain, device):
    """Copy a chain's tensor operands to `device` (same op list otherwise)."""
    out = []
    for kind, prm in chain:
        q = {}
        for k, v in prm.items():
            q[k] = v.to(device) if isinstance(v, torch.Tensor) else v
        out.append((kind, q))
    return out


def wl_chain(name, inp):
    """The tail chain of a named workload with its tensors bound from `inp`."""
    import kf_workloads
    wl = kf_workloads.WORKLOADS[name]
    chain = []
    for kind, prm in kf_workloads.chain_spec(wl):
        q = {}
        for k, v in prm.items():
            q[k] = inp[v] if (k in ("p0", "p1") and isinstance(v, str)) else v
        chain.append((kind, q))
    return chain
