"""The kernels' quantizer formulas, restated in C, against the oracle's code
functions on the CPU (Sec. 3 steps 2-3; readings r4, r10, r11): activation
codes on the Markstein path with the top clip taken on the input, the gather
kernel's calibrated variant (rounding by adding 1.5 * 2^23), and the weight
pack's estimate with its IEEE fallback near ties and for scales whose
RN(1/s) * 2^(n-1) overflows.  Every fp16 pattern (NaN and +-inf included) at
activation scales across [2^-60, 2^60], and weights on a grid of half-level
ties plus random values for scales from the smallest fp32 subnormal to FLT_MAX.
The GPU tests check the kernels themselves; this pins the formulas they use."""
import os
import subprocess
import tempfile

HERE = os.path.dirname(os.path.abspath(__file__))
ORACLE_C = os.path.join(os.path.dirname(HERE), "oracle", "soniq_oracle.c")


def test_quantizer_formulas_equal_the_oracle_codes():
    src = os.path.join(HERE, "csrc", "quantizer_check.c")
    with tempfile.TemporaryDirectory() as tmp:
        exe = os.path.join(tmp, "quantizer_check")
        subprocess.run(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", src, ORACLE_C,
                        "-o", exe, "-lm"], check=True)
        out = subprocess.run([exe], capture_output=True, text=True, check=True, timeout=600).stdout.split()
    bad_act, bad_gather, bad_w, cases = (int(x) for x in out)
    assert cases > 14 * 8 * 65536
    assert (bad_act, bad_gather, bad_w) == (0, 0, 0)
