"""The Python usage example of the package documentation: a whole ADPSGD run of resnet18-n8 on one GPU."""
import torch

from paper_2007_06134_gb300 import abi, inputs


def main():
    w = inputs.WORKLOADS["resnet18-n8"]                  # n = 8 replicas of a ResNet-18-sized vector
    h, c = inputs.problem(w)                             # the quadratic surrogate's curvatures and minimiser
    x = torch.empty((w.n, w.P), device="cuda")           # replicas, [n, P] fp32 in HBM
    v = torch.empty_like(x)                              # momentum buffers
    w0 = torch.zeros(w.P).pin_memory()                   # the initial model, on the host
    cfg = abi.make_config(w.n, w.P, momentum=w.mu, weight_decay=w.wd, noise_sigma=w.sigma, seed=w.seed,
                          fuse_sync_step=True)
    sched = abi.make_schedule(abi.ADPSGD, w.K, w.p_init, K_s=w.K_s, lr0=w.lr0, lr_factor=w.lr_factor,
                              milestones=w.milestones)   # Algorithm 2; abi.CPSGD for a constant period
    trace = abi.TraceBuffers(w.K)
    with abi.adpsgd_init(cfg, x, v, torch.from_numpy(h).cuda(), torch.from_numpy(c).cuda()) as ctx:
        abi.adpsgd_init_replicas(ctx, w0)                # every replica starts from w0, momentum 0
        stats = abi.adpsgd_run(ctx, sched, abi.adpsgd_state_init(sched), trace=trace)
    t = trace.arrays()                                   # per sync: k, p, S = Var[W_k], C2, loss
    print(stats.rounds, stats.equiv_period, stats.wire_bytes_per_node, t["p"][-1])
    return stats, t


if __name__ == "__main__":
    main()
