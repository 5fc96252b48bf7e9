"""GPU parity of the FOP injection through gated cross-attention adapters
(Sec. 3.2: the FOP tokens enter selected action-expert layers through gated
cross-attention adapters), through the C ABI, against the fp64 oracle.

Adapters every 2 layers (fp32 and bf16, ragged sizes, open gates so that the
adapters matter), and every layer at the pi0.5 width with one robot.
"""
import numpy as np
import pytest

import synth
from tests._harness import Case, check_step, gpu_session

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_34170_gb300 import build, load
    build.build()
    load()


def _open_gates(case, value=0.9):
    case.W = dict(case.W, a_gate=np.full_like(case.W["a_gate"], value))
    return case


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_adapters_every_second_layer(dtype):
    cfg = synth.ExpertConfig(layers=4, width=192, n_q_heads=6, n_kv_heads=2, head_dim=40, mlp_dim=320, slots=7,
                             action_dim=5, prefix=45, fop_tokens=3, batch=3, dtype=dtype, fop_adapter_every=2)
    case = _open_gates(Case(cfg))
    s = gpu_session(case)
    for i in range(3):
        check_step(case, s, label=f"{dtype} step {i}")
    s.close()


def test_adapters_pi05_width_one_robot():
    cfg = synth.PRESETS["pi05_bf16_b1"].replace(layers=4, fop_adapter_every=1)
    case = _open_gates(Case(cfg), 0.5)
    s = gpu_session(case)
    check_step(case, s, label="pi05 width, adapters in every layer")
    s.close()
