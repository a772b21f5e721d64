"""Comparison helpers shared by the parity tests (tolerances of the contract):
Philox words bit-exact; eps within 1e-5 * max(1, |eps|); fp32 parameters within
1e-5 relative plus the noise tolerance carried through the step
(1e-5 * sum_i |c_i| max(1, |eps_i|) for theta + sum_i c_i eps_i, which keeps
elements where theta and c eps cancel comparable); bf16 parameters within one
ulp, or, where theta and the noise term cancel so that one bf16 ulp is smaller
than that carried noise tolerance, within the tolerance plus one ulp."""
import numpy as np

EPS_TOL = 1e-5
F32_REL = 1e-5


def assert_eps_close(got, want, what=""):
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    err = np.abs(got - want)
    bound = EPS_TOL * np.maximum(1.0, np.abs(want))
    bad = np.nonzero(~(err <= bound))[0]
    assert bad.size == 0, (f"{what}: {bad.size} of {want.size} noise values out of tolerance; "
                           f"first at {bad[:5]}: got {got[bad[:5]]} want {want[bad[:5]]}")


def noise_abs_tol(eps_rows, coeffs):
    """1e-5 * sum_i |c_i| * max(1, |eps_i|): the eps tolerance carried through
    theta + sum_i c_i eps_i (eps_rows[i] is the oracle's eps of seed i)."""
    tol = 0.0
    for e, c in zip(eps_rows, coeffs):
        tol = tol + EPS_TOL * abs(float(c)) * np.maximum(1.0, np.abs(e))
    return tol


def assert_f32_close(got, want, what="", abs_tol=0.0):
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    err = np.abs(got - want)
    bound = F32_REL * np.abs(want) + abs_tol
    bad = np.nonzero(~(err <= bound))[0]
    assert bad.size == 0, (f"{what}: {bad.size} of {want.size} fp32 values out of tolerance; "
                           f"first at {bad[:5]}: got {got[bad[:5]]} want {want[bad[:5]]}")


def bf16_order(bits):
    """Map bf16 bit patterns to integers that step by one per representable value."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.int64)
    mag = b & 0x7FFF
    return np.where(b & 0x8000, -mag, mag)


def bf16_values(bits):
    """bf16 bit patterns (uint16) -> float64 values."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def assert_bf16_within_ulp(got_bits, want_bits, what="", ulps=1, abs_tol=0.0):
    d = np.abs(bf16_order(got_bits) - bf16_order(want_bits))
    g, w = bf16_values(got_bits), bf16_values(want_bits)
    ulp = 2.0 ** (np.floor(np.log2(np.maximum(np.maximum(np.abs(g), np.abs(w)), 2.0**-126))) - 7)
    near = np.abs(g - w) <= abs_tol + ulp
    bad = np.nonzero((d > ulps) & ~near)[0]
    assert bad.size == 0, (f"{what}: {bad.size} of {d.size} bf16 values more than {ulps} ulp "
                           f"apart; first at {bad[:5]}: got {np.asarray(got_bits)[bad[:5]]} "
                           f"want {np.asarray(want_bits)[bad[:5]]}")


def build_c_consumer(out_dir):
    """Compiles tests/abi_c_consumer.c (C99) against include/esopt.h and links
    it to the in-tree libesopt.so and the CUDA runtime. Returns the path of
    the executable."""
    import glob
    import os
    import subprocess
    here = os.path.dirname(os.path.abspath(__file__))
    root = os.path.dirname(here)
    cuda = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    libdirs = [d for d in [os.path.join(cuda, "lib64")] + glob.glob(os.path.join(cuda, "targets", "*", "lib"))
               if glob.glob(os.path.join(d, "libcudart.so*"))]
    if not libdirs:
        raise RuntimeError("libcudart.so not found under " + cuda)
    build = os.path.join(root, "paper_2608_17310_gb300", "_build")
    exe = os.path.join(str(out_dir), "abi_c_consumer")
    cmd = ["gcc", "-std=c99", "-Wall", "-Wextra", "-Werror",
           f"-I{os.path.join(root, 'include')}", f"-I{os.path.join(cuda, 'include')}",
           os.path.join(here, "abi_c_consumer.c"), "-o", exe,
           f"-L{build}", "-lesopt", f"-L{libdirs[0]}", "-lcudart",
           f"-Wl,-rpath,{build}", f"-Wl,-rpath,{libdirs[0]}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("building the C consumer failed:\n" + r.stderr)
    return exe
