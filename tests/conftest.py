import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long-running")


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """The worst value error each parity check observed against the oracle:
    relative error for binary32 outputs, bfloat16 ulps for bfloat16 outputs,
    and the entries that needed the cancellation bound of parity_util."""
    tr = terminalreporter
    opt = getattr(sys.modules.get("test_gpu_optimizer"), "WORST_OPT", None)
    if opt:
        tr.section("ISO-Optimizer step: worst error / derived bound")
        for what, ratio in sorted(opt.items()):
            tr.write_line(f"{what}: " + ", ".join(f"{k} {v:.3g}" for k, v in ratio.items()))
    frame = getattr(sys.modules.get("test_gpu_frame"), "WORST_FRAME", None)
    if frame:
        tr.section("frame-space merge: worst error / derived bound")
        for what, ratio in sorted(frame.items()):
            tr.write_line(f"{what}: " + ", ".join(f"{k} {v:.3g}" for k, v in ratio.items()))
    try:
        from parity_util import WORST
    except ImportError:
        return
    if not WORST:
        return
    tr.section("worst observed value error against the oracle")
    for what, (worst, n, n_cancel, kind) in sorted(WORST.items()):
        unit = "ulp (bf16)" if kind == "ulp" else "relative (f32)"
        tr.write_line(f"{what}: {worst:.3g} {unit} over {n} entries; "
                      f"{n_cancel} on the cancellation bound")
