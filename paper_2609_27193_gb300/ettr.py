"""Effective training time ratio under repeated failures (§4.5).

ETTR (Eq. 15) is the fraction of wall-clock time spent on useful training:
t_train / (t_train + t_ckpt + t_recovery), where a recovery costs
t_load + t_retrain + t_reconstruct (Eq. 13).  Failures arrive as a Poisson
process with mean time between failures MTBF while the job runs.

A checkpointing policy is described by the segment between two durable
checkpoints: `k` iterations of t_iter each plus the checkpoint time that
blocks training in that segment.  Work is lost back to the last durable
checkpoint.  `simulate` injects failures event by event and accounts every
component of Eq. 13-15; `expected_ettr` is the exact expectation for the
same process (a segment of wall length S completes after an expected
(e^{S/MTBF} - 1) (MTBF + R) seconds when each failure costs R to recover).

This is a CPU model, fed with the costs the GPU path measures (bench.py
JSON): the device time of the checkpoint step, the device->host leg, and
the host->device restore of the composite.
"""
import argparse
import json
import math
import random
from dataclasses import dataclass, field


@dataclass
class Policy:
    name: str
    t_iter: float            # seconds of training per iteration
    k: int                   # iterations between durable checkpoints
    t_ckpt_segment: float    # checkpoint seconds that block training, per segment
    t_load: float            # seconds to read the restart state back
    t_reconstruct: float = 0.0
    t_restart: float = 0.0   # fixed cost of a restart (process, scheduler)

    @property
    def segment(self):
        return self.k * self.t_iter + self.t_ckpt_segment

    @property
    def recovery(self):
        return self.t_load + self.t_reconstruct + self.t_restart


def expected_ettr(p, mtbf):
    """Exact ETTR of the failure process for policy p (seconds, MTBF > 0)."""
    if math.isinf(mtbf):
        return p.k * p.t_iter / p.segment
    lam = 1.0 / mtbf
    expected_segment = math.expm1(lam * p.segment) * (mtbf + p.recovery)
    return p.k * p.t_iter / expected_segment


@dataclass
class Tally:
    train: float = 0.0        # useful iterations' time (kept work)
    ckpt: float = 0.0         # blocking checkpoint time of completed segments
    load: float = 0.0
    reconstruct: float = 0.0
    restart: float = 0.0
    retrain: float = 0.0      # work (and checkpoint time) lost to failures
    failures: int = 0
    extra: dict = field(default_factory=dict)

    @property
    def wall(self):
        return self.train + self.ckpt + self.load + self.reconstruct + self.restart + self.retrain

    @property
    def ettr(self):
        return self.train / self.wall if self.wall > 0 else 1.0


def simulate(p, mtbf, total_iters, seed=0):
    """Event-driven run of `total_iters` iterations with Poisson failures of
    mean `mtbf` seconds; returns the tally of Eq. 13-15's components."""
    rng = random.Random(seed)
    lam = 0.0 if math.isinf(mtbf) else 1.0 / mtbf
    next_failure = rng.expovariate(lam) if lam > 0 else math.inf
    clock = 0.0
    done = 0
    t = Tally()
    while done < total_iters:
        k = min(p.k, total_iters - done)
        seg = k * p.t_iter + (p.t_ckpt_segment if k == p.k else p.t_ckpt_segment * k / p.k)
        if clock + seg <= next_failure:
            clock += seg
            done += k
            t.train += k * p.t_iter
            t.ckpt += seg - k * p.t_iter
            continue
        # failure inside the segment: its work is lost, then the job recovers
        lost = next_failure - clock
        t.retrain += lost
        t.load += p.t_load
        t.reconstruct += p.t_reconstruct
        t.restart += p.t_restart
        t.failures += 1
        clock = next_failure + p.recovery
        next_failure = clock + rng.expovariate(lam)
    return t


def young_daly_k(t_iter, t_ckpt_full, mtbf):
    """Checkpoint interval (iterations) near the optimum sqrt(2 C MTBF) for a
    full checkpoint of blocking cost C."""
    return max(1, int(round(math.sqrt(2.0 * t_ckpt_full * mtbf) / t_iter)))


def policies_from_bench(line, t_iter, h2d_gbps=None, restart=0.0, d2h_overlaps=True):
    """LayerCheck vs full-state checkpoint policies from a bench.py JSON line.

    LayerCheck checkpoints every iteration: its blocking time is the device
    step (measure + select + pack); the D2H of the persisted layers overlaps
    the next iteration when it is shorter than t_iter (else the excess
    blocks).  A full checkpoint moves the whole state (every layer every
    time) over the same link.  Both restart by reading the full state."""
    persisted = line["persisted_bytes_per_step"]
    link = (line.get("e2e") or {}).get("d2h_link_GBps_measured") or 193.0
    # every layer's block (the bench reports it; older lines: estimated from
    # the persisted share of the layers)
    full_bytes = line.get("full_state_bytes") or persisted / max(line["selected_fraction"], 1e-9)
    step_s = line["ms_per_step"] / 1e3
    d2h_s = persisted / (link * 1e9)
    # the D2H hides behind the next iteration up to t_iter when it overlaps
    hidden = min(d2h_s, t_iter) if d2h_overlaps else 0.0
    lc_block = step_s + (d2h_s - hidden)
    full_d2h = full_bytes / (link * 1e9)
    load = full_bytes / ((h2d_gbps or link) * 1e9)
    return {
        "layercheck": Policy("layercheck (every iteration)", t_iter, 1, lc_block, load, 0.0, restart),
        "full_every_iter": Policy("full state every iteration", t_iter, 1, full_d2h, load, 0.0, restart),
        "full_d2h": full_d2h,
        "load": load,
    }


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--bench", required=True, help="a bench.py JSON line (file)")
    ap.add_argument("--t-iter", type=float, required=True, help="training seconds per iteration")
    ap.add_argument("--h2d-gbps", type=float, default=None)
    ap.add_argument("--restart", type=float, default=30.0, help="fixed restart seconds")
    ap.add_argument("--mtbf-hours", type=float, nargs="+", default=[0.01, 0.1, 0.5, 1.0, 3.0])
    args = ap.parse_args()
    line = json.loads(open(args.bench).read().strip().splitlines()[-1])
    pol = policies_from_bench(line, args.t_iter, args.h2d_gbps, args.restart)
    rows = []
    for h in args.mtbf_hours:
        mtbf = h * 3600.0
        k = young_daly_k(args.t_iter, pol["full_d2h"], mtbf)
        periodic = Policy("full state every %d iterations" % k, args.t_iter, k, pol["full_d2h"],
                          pol["load"], 0.0, args.restart)
        rows.append({"mtbf_h": h,
                     "layercheck": expected_ettr(pol["layercheck"], mtbf),
                     "full_every_iter": expected_ettr(pol["full_every_iter"], mtbf),
                     "full_periodic_k": k,
                     "full_periodic": expected_ettr(periodic, mtbf)})
    print(json.dumps(rows, indent=1))


if __name__ == "__main__":
    main()
