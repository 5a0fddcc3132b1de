"""The two attention kernels for fp16-carried q|k|v with dh = 64: the tensor-memory kernel (tcgen05
MMAs, TMEM accumulators, TMA key stream; the default) and the warp-MMA kernel it replaces
(selected for every problem by ILWDETR_ATTENTION_TC=0, read once per process).  Each is compared
with the oracle; the warp-MMA run happens in a child process so that the setting takes effect."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("setting", ["1", "0"])
def test_attention_kernels_match_oracle(setting):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    env = dict(os.environ, ILWDETR_ATTENTION_TC=setting)
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_gpu_parity.py"), "-k",
                        "test_attention and f16 or test_attention_f16_output or block_forward"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-2000:]
    assert " passed" in r.stdout
