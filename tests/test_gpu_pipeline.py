"""The chunked host pipeline (profiles in pinned host memory) gives exactly the
device-resident path's results, for every chunking including ragged ones."""
import numpy as np
import pytest

import oracle
from paper_2101_07968_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dc():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_07968_gb300 import build, dynacomm
    build.build()
    dynacomm.lib()
    return dynacomm


@pytest.mark.parametrize("name,batch,chunks", [("vgg16", 50_003, 7), ("resnet50", 4_097, 3),
                                               ("tiny", 100, 1), ("alexnet", 33, 40)])
def test_host_pipeline_matches_oracle(dc, name, batch, chunks):
    import torch
    cfg = wl.with_batch(wl.config(name), batch)
    ref = oracle.profile_gen(cfg)
    host_in = {k: torch.from_numpy(v).pin_memory() for k, v in ref.items()}
    pipe = dc.HostPipeline(batch, cfg["L"], chunks=chunks)
    host_out = pipe.host_buffers()
    for _ in range(2):  # twice: buffers and workspace are reused
        pipe.run(host_in, host_out)
        torch.cuda.synchronize()
        W = dc.words(cfg["L"])
        for d, (c, x) in ((dc.FWD, ("fc", "pt")), (dc.BWD, ("bc", "gt"))):
            exp = oracle.schedule_batch(d, ref[c], ref[x], ref["dt"], nthreads=8)
            assert np.array_equal(host_out[(d, "makespan")].numpy(), exp["makespan"])
            assert np.array_equal(host_out[(d, "nseg")].numpy(), exp["nseg"])
            assert np.array_equal(host_out[(d, "bits")].numpy().view(np.uint32)[:, :W],
                                  exp["bits"])
            assert np.array_equal(host_out[(d, "replay")].numpy(), exp["makespan"])


def test_host_pipeline_shared_transfer_buffer(dc):
    """gt passed as the pt host buffer (equal transfer costs): copied once, the
    same results as separate buffers."""
    import torch
    cfg = wl.with_batch(wl.config("vgg16"), 20_011)
    ref = oracle.profile_gen(cfg)
    assert np.array_equal(ref["pt"], ref["gt"])
    sep = {k: torch.from_numpy(v).pin_memory() for k, v in ref.items()}
    shared = dict(sep)
    shared["gt"] = shared["pt"]
    pipe = dc.HostPipeline(cfg["batch"], cfg["L"], chunks=5)
    out_sep, out_shared = pipe.host_buffers(), pipe.host_buffers()
    pipe.run(sep, out_sep)
    torch.cuda.synchronize()
    pipe.run(shared, out_shared)
    torch.cuda.synchronize()
    for k in out_sep:
        assert torch.equal(out_sep[k], out_shared[k]), k
    h_sep, _ = pipe.bytes_per_run(sep)
    h_shared, _ = pipe.bytes_per_run(shared)
    assert h_sep - h_shared == ref["gt"].nbytes
