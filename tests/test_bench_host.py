"""Host-side logic of bench.py (no GPU): an extra row that fails is reported in the JSON line and
does not take the headline measurement down with it."""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_failing_extra_is_reported_and_the_others_kept():
    result = {"metric": "m", "value": 1.0}

    def ok():
        return {"row_a": {"GB_s": 1.0}}

    def broken():
        raise RuntimeError("device error in the measurement")

    bench._extra(result, "a", ok)
    bench._extra(result, "b", broken)
    assert result["row_a"] == {"GB_s": 1.0}
    assert result["value"] == 1.0
    assert "RuntimeError: device error" in result["extra_errors"]["b"]
    json.dumps(result)  # still one JSON line
