"""Run the sketching step (forward with lse, then backward) a few times on a
sub-batch of one of the evaluation workloads, for kernel profiling.

    python -m paper_2609_08443_gb300.profile_case --config 4 --users 4 --steps 2

The sub-batch keeps the per-user shapes of the workload (e.g. 100000 tokens per
user, H=8, d=128, P=512 for config 4) so the kernels see the same tiles; its
K and V still exceed L2 (4 users of config 4: 1.6 GB), while the whole run
holds only a few GB on the device.
"""
from __future__ import annotations

import argparse

import torch

from . import binding, workloads as wl


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--config", type=int, default=4)
    ap.add_argument("--users", type=int, default=4)
    ap.add_argument("--steps", type=int, default=2)
    ap.add_argument("--fwd-only", action="store_true")
    ap.add_argument("--tokenwise", action="store_true", help="token-wise normalisation (Sec. 5.1) instead")
    args = ap.parse_args()
    spec = wl.config(args.config)
    sub = wl.sub_spec(spec, list(range(min(args.users, spec.B if spec.kind != "extremes" else 4100))))
    dev = torch.device("cuda", 0)
    data = wl.make_device(sub, dev)
    K, V, Q, cu, dS = data["K"], data["V"], data["Q"], data["cu_seqlens"], data["dsketch"]
    for _ in range(args.steps):
        if args.tokenwise:
            s, lse = binding.sa_sketch_fwd_tokenwise(K, V, cu, Q, sub.scale, want_lse=True)
            if not args.fwd_only and spec.bwd:
                binding.sa_sketch_bwd_tokenwise(K, V, cu, Q, dS, sub.scale, sketch=s, lse=lse)
            continue
        s, lse = binding.sa_sketch_fwd(K, V, cu, Q, sub.scale, want_lse=True)
        if not args.fwd_only and spec.bwd:
            binding.sa_sketch_bwd(K, V, cu, Q, dS, sub.scale, lse=lse)
    torch.cuda.synchronize()
    print("ok", binding.sa_main_kernel_name(sub.P, sub.d, binding.SA_BF16, False),
          binding.sa_main_kernel_name(sub.P, sub.d, binding.SA_BF16, True))


if __name__ == "__main__":
    main()
