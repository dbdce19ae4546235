import json
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running on CPU")


def pytest_collection_modifyitems(config, items):
    # Keep file order (pytest default), but make sure files named test_zz_*
    # run after everything else even if collected from several directories.
    items.sort(key=lambda it: os.path.basename(str(it.fspath)).startswith("test_zz_"))


def pytest_terminal_summary(terminalreporter):
    """Prints the figures the GPU parity tests report (gpu_util.REPORT) and,
    if DLM_TEST_REPORT names a file, writes them there as JSON."""
    gu = sys.modules.get("gpu_util")
    if gu is None or not any(gu.REPORT.values()):
        return
    tr = terminalreporter
    errs = gu.REPORT["attention_errors"]
    if errs:
        tr.write_sep("-", f"attention error statistics ({len(errs)} comparisons)")
        for e in errs:
            tr.write_line(f"{e['dtype']:4s} max_abs {e['max_abs']:.3e}  max_abs/max|ref| {e['max_rel']:.3e}  "
                          f"mean_abs {e['mean_abs']:.3e}  mean_abs/mean|ref| {e['mean_rel']:.3e}  "
                          f"bias/mean|ref| {e['bias_rel']:+.2e}  max|ref| {e['max_ref']:.3g}  {e['where']}")
    mar = gu.REPORT["margin_limited"]
    if mar:
        tr.write_sep("-", "decision-margin protocol: positions left out of the exact update comparison")
        for m in mar:
            tr.write_line(f"{m['positions']:6d} of {m['checked']:8d} (differing {m['differing']})  {m['where']}")
    for n in gu.REPORT.get("notes", []):
        tr.write_line(n["text"])
    path = os.environ.get("DLM_TEST_REPORT")
    if path:
        with open(path, "w") as f:
            json.dump(gu.REPORT, f, indent=1)
