"""Host-side logic that needs no GPU: the bench's choice of the binding roof and
the host pipeline's detection of inputs that share one buffer."""
import numpy as np
import torch

import bench
from paper_2101_07968_gb300 import dynacomm as dc


def test_binding_roof_takes_the_larger_fraction():
    alu = {"bound": "alu", "frac": 0.52, "achieved": 7.0, "peak": 13.4}
    hbm = {"bound": "hbm", "frac": 0.42, "achieved": 2860.0, "peak": 6784.8}
    r = bench.binding_roof(alu, hbm, kernel="k", traffic=None)
    assert r["bound"] == "alu" and r["frac"] == 0.52 and r["kernel"] == "k"
    assert r["other_roof"]["bound"] == "hbm" and r["traffic"] is None
    # a memory-bound pass (L = 8): the HBM roof binds
    alu["frac"], hbm["frac"] = 0.18, 0.59
    r = bench.binding_roof(alu, hbm)
    assert r["bound"] == "hbm" and r["other_roof"]["bound"] == "alu"


def test_shared_inputs_by_buffer_not_by_value():
    keys = ("fc", "pt", "bc", "gt", "dt")
    a = torch.arange(12, dtype=torch.int64).reshape(3, 4)
    same_values = a.clone()
    host = {"fc": a, "pt": same_values, "bc": torch.zeros(3, 4, dtype=torch.int64),
            "gt": same_values, "dt": torch.zeros(3, dtype=torch.int64)}
    canon = dc.shared_inputs(host, keys)
    assert canon == {"fc": "fc", "pt": "pt", "bc": "bc", "gt": "pt", "dt": "dt"}
    # equal contents in distinct buffers are copied separately
    host["gt"] = same_values.clone()
    assert dc.shared_inputs(host, keys)["gt"] == "gt"
    # a view of a different size over the same start is a different input
    host["gt"] = a.reshape(-1)[:4]
    assert dc.shared_inputs(host, keys)["gt"] == "gt"
    assert dc.shared_inputs(None, keys) == {k: k for k in keys}
    assert np.array_equal(a.numpy(), same_values.numpy())
