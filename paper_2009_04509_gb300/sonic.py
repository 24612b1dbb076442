"""Scale-out latency model of the paper's as-a-service setup (Sec. 3.3,
Eqs. 1-5), as plain host functions.

A CPU job of t_cpu seconds has a fraction p that is offloaded.  With the GPU
always available, the job takes

    t_ideal = (1 - p) t_cpu + t_gpu + t_latency                    (Eq. 2)

where t_latency = t_preproc + t_transmit + t_travel is the extra latency of
the service (preprocessing on the CPU, sending the inputs, round trips).  The
GPU saturates once more CPU jobs share it than one job's time can cover:

    n_cpu / n_gpu > t_ideal / t_gpu                                (Eq. 3)

and the job time becomes

    t_sonic = (1 - p) t_cpu + t_gpu [1 + max(0, n_cpu/n_gpu - t_ideal/t_gpu)]
              + t_latency                                          (Eq. 4)

which reduces to t_gpu n_cpu / n_gpu when saturated (Eq. 5).  The break-even
ratio t_ideal / t_gpu is the number of CPU jobs one GPU can serve.

The paper's inputs (Sec. 3.3): t_cpu = 330 s, p = 0.65, t_preproc = 7 s,
t_transmit = 2.05-4.1 s (4.1 Gbit per event over 1-2 Gbps), t_travel = 0.38 s
(32 requests of 12 ms, large batch) or 2.6 s (214 requests, small batch), and
t_gpu = 1.77 s (55,000 inferences at 31,000 per second) or 2.5 s.
"""
from __future__ import annotations

from dataclasses import dataclass

PAPER_T_CPU = 330.0          # s, CPU-only job (Sec. 3.1 / 3.3)
PAPER_P = 0.65               # accelerated fraction
PAPER_T_PREPROC = 7.0        # s
PAPER_T_TRANSMIT = (2.05, 4.1)  # s, 2 Gbps / 1 Gbps
PAPER_T_TRAVEL_LARGE = 0.38  # s, 32 requests x 12 ms
PAPER_T_TRAVEL_SMALL = 2.6   # s
PAPER_INFERENCES = 55_000    # patches per event
PAPER_GPU_RATE = (31_000.0, 22_000.0)  # inferences per second per GPU: with / without dynamic batching


@dataclass(frozen=True)
class Job:
    t_cpu: float
    p: float
    t_gpu: float
    t_preproc: float = 0.0
    t_transmit: float = 0.0
    t_travel: float = 0.0

    @property
    def t_latency(self) -> float:
        return self.t_preproc + self.t_transmit + self.t_travel


def t_ideal(job: Job) -> float:
    """Job time with the GPU always available (Eq. 2)."""
    return (1.0 - job.p) * job.t_cpu + job.t_gpu + job.t_latency


def saturated(job: Job, n_cpu: float, n_gpu: float) -> bool:
    """The GPU saturation condition (Eq. 3)."""
    return n_cpu / n_gpu > t_ideal(job) / job.t_gpu


def t_sonic(job: Job, n_cpu: float, n_gpu: float) -> float:
    """Job time with n_cpu jobs sharing n_gpu GPUs (Eq. 4)."""
    excess = max(0.0, n_cpu / n_gpu - t_ideal(job) / job.t_gpu)
    return (1.0 - job.p) * job.t_cpu + job.t_gpu * (1.0 + excess) + job.t_latency


def cpu_per_gpu(job: Job) -> float:
    """CPU jobs one GPU serves before it saturates: t_ideal / t_gpu."""
    return t_ideal(job) / job.t_gpu


def paper_job(dynamic_batching: bool = True, link_gbps: float = 2.0, large_batch: bool = True) -> Job:
    """The paper's job with its measured inputs."""
    rate = PAPER_GPU_RATE[0] if dynamic_batching else PAPER_GPU_RATE[1]
    transmit = PAPER_T_TRANSMIT[0] if link_gbps >= 2.0 else PAPER_T_TRANSMIT[1]
    return Job(t_cpu=PAPER_T_CPU, p=PAPER_P, t_gpu=PAPER_INFERENCES / rate, t_preproc=PAPER_T_PREPROC,
               t_transmit=transmit, t_travel=PAPER_T_TRAVEL_LARGE if large_batch else PAPER_T_TRAVEL_SMALL)


def gb300_job(hits_per_s: float, inferences: int = PAPER_INFERENCES, t_cpu: float = PAPER_T_CPU,
              p: float = PAPER_P) -> Job:
    """The paper's CPU job with its offloaded part replaced by this library's
    measured throughput.  ``hits_per_s`` must be an end-to-end figure, taken
    through the call with host buffers (the planes and hits copied to the
    device, the scores copied back), so that the host-device copies are
    inside t_gpu; the patch cut runs on the GPU (no CPU preprocessing) and, in
    one process, there is no network transfer or round trip."""
    return Job(t_cpu=t_cpu, p=p, t_gpu=inferences / hits_per_s)
