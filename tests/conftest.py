import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


def pytest_terminal_summary(terminalreporter):
    """Element-wise error diagnostics of the GPU forwards checked in the run."""
    mod = sys.modules.get("test_gpu_parity") or sys.modules.get("tests.test_gpu_parity")
    diag = getattr(mod, "DIAG", None) if mod else None
    if not diag:
        return
    tr = terminalreporter
    tr.section("element-wise |y - ref| / max(|ref|, 1e-3 rms(ref)) (per forward checked)")
    worst = max(d[1] for d in diag)
    tr.write_line(f"{len(diag)} forwards; worst per-tensor max|y - ref| / max|ref| = {worst:.3e}")
    tr.write_line(f"median of the element-wise medians = "
                  f"{sorted(d[2]['p50'] for d in diag)[len(diag) // 2]:.3e}; "
                  f"largest element-wise median = {max(d[2]['p50'] for d in diag):.3e}")
    for name, err, ew in diag:
        tr.write_line(f"  {name}: tensor {err:.2e}  elem p50 {ew['p50']:.2e} "
                      f"p99 {ew['p99']:.2e} max {ew['max']:.2e}")
