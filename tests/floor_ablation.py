"""Which of the CUDA path's bf16 rounding points set the full-depth error
floor (a diagnostic on the CPU, not a test).

The fp64 emulation of the CUDA path's storage formats (tests/bf16_emulation.py,
pinned by tests/test_bf16_emulation.py) runs every sample of the chosen
samples through all blocks alongside the fp64 oracle (oracle.model), once
with every rounding point, once with each point left out, and once with
each main point alone (plus the fp32 residual stream), and prints each
configuration's max |err| / rms of the pooled features against the oracle
every few blocks.  The weights and inputs are the seeded synthetic ones of
the workload (CPU generator).

    python tests/floor_ablation.py --workload llama7b --tenant 30 --samples 1

The 7B-class run (one ~330-token sample, 32 blocks) holds about 16 GB of
host memory and takes about 15 minutes on 8 cores.
"""
import argparse
import sys
import time
from pathlib import Path

sys.path.insert(0, str(Path(__file__).resolve().parents[1]))

import synth  # noqa: E402
from oracle import model as M  # noqa: E402
from tests import bf16_emulation as E  # noqa: E402
from tests.gpu_helpers import tenant_samples  # noqa: E402
from tests.helpers import rel_err  # noqa: E402

MAIN_POINTS = ("norm", "qkv", "p", "attn_out", "u")


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--workload", default="llama7b")
    ap.add_argument("--tenant", type=int, default=30)
    ap.add_argument("--samples", type=int, default=1, help="first N samples of the tenant")
    ap.add_argument("--every", type=int, default=4, help="print every N blocks")
    args = ap.parse_args()

    w = synth.make_workload(args.workload)
    bw = synth.to_numpy_tree(synth.make_backbone_weights(w))
    inp = synth.to_numpy_tree(synth.make_inputs(w))
    bb = M.backbone_dict(w)
    smp = tenant_samples(w, args.tenant)[:args.samples]
    xs = [M.sample_embeddings(bb, vars(s), inp["vision"], inp["text_ids"], bw["text_table"])
          for s in smp]
    tn = [args.tenant] * len(xs)
    configs = {"all": E.ALL}
    for p in E.ALL:
        configs["all but " + p] = tuple(q for q in E.ALL if q != p)
    for p in MAIN_POINTS:
        configs[p + " alone"] = (p, "resid")
    emus = {k: E.Emulation(w.backbone, xs, tn, r) for k, r in configs.items()}
    ref = list(xs)
    fin = bw["final_norm"]
    t0 = time.time()
    n = len(bw["layers"])
    for li, lw in enumerate(bw["layers"]):
        wl = E.widen_layer(lw)
        ref = [M.block(bb, wl, x, t) for x, t in zip(ref, tn)]
        for e in emus.values():
            e.block(wl)
        if (li + 1) % args.every == 0 or li + 1 == n:
            rp = [M.mean_pool(M.rmsnorm(x, fin, bb["eps"])) for x in ref]
            errs = {k: max(rel_err(p, r) for p, r in zip(e.pooled(fin), rp))
                    for k, e in emus.items()}
            print(f"blocks {li + 1} ({time.time() - t0:.0f} s): " +
                  ", ".join(f"{k} {v:.4f}" for k, v in errs.items()), flush=True)


if __name__ == "__main__":
    main()
