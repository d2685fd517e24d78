import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running CPU test")


def pytest_collection_modifyitems(config, items):
    try:
        import torch
        has_gpu = torch.cuda.is_available()
    except Exception:  # pragma: no cover
        has_gpu = False
    if has_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Per-key selection parity at a glance: how many (unit, KV head)
    selections were compared with the oracle, how many keys differed from the
    oracle's kept set, and how wide the cutoff bands were."""
    parity = sys.modules.get("tests.parity")
    if parity is None:
        return
    plog = getattr(parity, "PROXY_LOG", None)
    if plog:
        nd = sum(n for _, n, _ in plog)
        tot = sum(t for _, _, t in plog)
        terminalreporter.write_line(
            f"proxy parity (level A): {len(plog)} comparisons, {nd} of {tot} bf16 elements "
            f"differ from the oracle's ({nd / max(tot, 1):.2e})")
    log = getattr(parity, "SELECTION_LOG", None)
    if not log:
        return
    n = len(log)
    mism = sum(m for _, m, _ in log)
    with_mism = [(w, m, b) for w, m, b in log if m]
    band = max(b for _, _, b in log)
    tr = terminalreporter
    tr.write_line(f"selection parity: {n} (unit, KV head) selections checked per key; "
                  f"{mism} keys differ from the oracle's kept sets in {len(with_mism)} of them; "
                  f"widest cutoff band {band} keys")
    for w, m, b in with_mism[:20]:
        tr.write_line(f"  {w}: {m} keys differ, {b} keys in the cutoff band")
