"""The activation kernels form a / s by one Markstein correction step on
RN(1 / s) instead of a division (Sec. 3 step 2 fixes the quotient; reading c2:
the correctly rounded fp32 quotient).  This CPU test checks, exhaustively over
every finite fp16 input and every positive finite fp16 scale plus seeded random
fp32 scales in [2^-60, 2^60], that the two are the same fp32 value, so the
codes the kernels decide are the ones the oracle's IEEE division decides; and
that the corrected quotient of s by itself is exactly 1 (a calibrated scale
clips larger inputs, +inf among them, to s before the quotient)."""
import os
import subprocess
import tempfile

HERE = os.path.dirname(os.path.abspath(__file__))


def test_markstein_quotient_equals_ieee_division_for_every_fp16_input():
    src = os.path.join(HERE, "csrc", "markstein_check.c")
    with tempfile.TemporaryDirectory() as tmp:
        exe = os.path.join(tmp, "markstein_check")
        subprocess.run(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", src, "-o", exe, "-lm"],
                       check=True)
        out = subprocess.run([exe, "4000"], capture_output=True, text=True, check=True, timeout=900).stdout.split()
    bad, scales, inputs = (int(x) for x in out)
    assert inputs == 63488                      # every finite fp16 pattern
    assert scales > 31743 + 3900                # all positive finite fp16 scales and the random ones
    assert bad == 0
