"""The handoff workload driven from C (cdriver/handoff_step.c) through the C
ABI alone: a small run whose copied outputs all hold their inputs' bytes."""
import json
import subprocess

import pytest

pytestmark = pytest.mark.gpu


def test_c_driver_small_handoff(lib):
    from paper_2607_26566_gb300 import build as b

    exe = b.build_cdriver()
    # B=1, 8 requests on 2 streams, 3 steps after 1 warm-up, 2 MiB pages, 1 GiB pool
    out = subprocess.run([exe, "1", "8", "2", "3", "1", str(2 << 20), "1"], capture_output=True, text=True,
                         timeout=300)
    assert out.returncode == 0, out.stderr
    d = json.loads(out.stdout.strip().splitlines()[-1])
    assert d["outputs_ok"] is True
    assert d["B"] == 1 and d["requests"] == 8 and d["streams"] == 2 and d["gbs"] > 0
