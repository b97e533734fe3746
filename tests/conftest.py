import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built libpbd")
    config.addinivalue_line("markers", "slow: full-size model on the CPU oracle (seconds to minutes)")


@pytest.fixture(scope="session")
def tiny():
    """Tiny Qwen3-style shape with seeded base weights, adapter and a 64-token prompt."""
    from paper_2607_12422_gb300 import synth
    import oracle
    S = synth.TINY
    base = synth.gen_base_weights(S)
    ad = synth.gen_adapter(S)
    prompt = synth.gen_prompts(S, [64])[0]
    return dict(shape=S, base=base, adapter=ad, prompt=prompt, model=oracle.OracleModel(S, base, ad))


@pytest.fixture(scope="session")
def tiny_zeroB():
    """Same tiny model with the adapter's B matrices zeroed (the LoRA delta vanishes)."""
    from paper_2607_12422_gb300 import synth
    import oracle
    S = synth.TINY
    base = synth.gen_base_weights(S)
    ad = synth.gen_adapter(S, zero_B=True)
    prompt = synth.gen_prompts(S, [64])[0]
    return dict(shape=S, base=base, adapter=ad, prompt=prompt, model=oracle.OracleModel(S, base, ad))


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """The measured GPU-vs-oracle logit differences and near-ties of the parity tests that ran."""
    import _parity
    lines = _parity.summary_lines()
    if not lines:
        return
    terminalreporter.write_sep("-", "parity measurements")
    for line in lines:
        terminalreporter.write_line(line)
    path = os.environ.get("PBD_PARITY_JSON")
    if path:
        import json
        with open(path, "w") as f:
            json.dump(_parity.RECORDS, f, indent=1)
