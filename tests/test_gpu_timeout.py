"""A bounded pipeline wait that runs out: failure detection without a GPU fault.

Every wait inside the tensor-core kernels gives up after a time limit.  The
kernel then stops all its roles, drains the copies and tensor-core work still
in flight, frees its tensor memory, records SA_ERR_TIMEOUT in the call's
workspace, and the call's later kernels skip their work.  The limit is 2 s;
no correct pipeline comes near it.  This test lowers it to 1 ns so that waits
run out, checks the reported status, restores the limit and checks that the
next call on the same device and workspace is bitwise the same as before.
"""
import pytest
import torch

from paper_2609_08443_gb300 import binding, workloads as wl

pytestmark = pytest.mark.gpu

SA_ERR_TIMEOUT = 5


@pytest.mark.parametrize("P,d", [(256, 64), (512, 128)], ids=["fused", "cluster-pair"])
def test_wait_timeout_is_reported_and_the_next_call_is_clean(cuda_lib, P, d):
    assert binding.sa_main_kernel_name(P, d, binding.SA_BF16, False).startswith("tc")
    # about 16 tiles per worker at P = 256 (32 per cluster pair at P = 512), so the pipelines wait
    spec = wl.custom([70000, 3000, 0, 81000], H=2, P=P, d=d, dtype=wl.BF16, seed=31, bwd=False)
    t = wl.host_to_torch(spec, wl.make_host(spec), torch.device("cuda"))
    N, H, d = t["K"].shape
    B = t["cu_seqlens"].numel() - 1
    ws = torch.empty(binding.sa_workspace_size(B, N, H, spec.P, d, binding.SA_BF16, 0), dtype=torch.uint8,
                     device="cuda")

    def fwd():
        return binding.sa_sketch_fwd(t["K"], t["V"], t["cu_seqlens"], t["Q"], spec.scale, want_lse=True, ws=ws)

    ref, ref_lse = (x.clone() for x in fwd())
    assert binding.sa_get_device_error(ws) == 0
    statuses = []
    try:
        binding.sa_set_wait_limit_ns(1)
        for _ in range(3):
            fwd()
            statuses.append(binding.sa_get_device_error(ws))
            if statuses[-1] == SA_ERR_TIMEOUT:
                break
    finally:
        binding.sa_set_wait_limit_ns(0)  # back to the default limit
    assert SA_ERR_TIMEOUT in statuses, statuses
    sketch, lse = fwd()
    assert binding.sa_get_device_error(ws) == 0
    torch.cuda.synchronize()
    assert torch.equal(sketch, ref) and torch.equal(lse, ref_lse)
