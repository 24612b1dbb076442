"""The scale-out latency model (Sec. 3.3, Eqs. 2-5) against the paper's own
figures and the model's algebra."""
import math

import pytest

from paper_2009_04509_gb300 import sonic


def test_paper_inputs_give_the_paper_terms():
    job = sonic.paper_job(dynamic_batching=True, link_gbps=2.0, large_batch=True)
    assert job.t_gpu == pytest.approx(1.77, abs=0.005)  # 55,000 / 31,000 s
    assert sonic.paper_job(dynamic_batching=False).t_gpu == pytest.approx(2.5, abs=0.005)
    assert job.p * job.t_cpu == pytest.approx(214.5)  # the 220 s module minus preprocessing, about
    # the transmit bound: 4.1 Gbit over 2 and 1 Gbps
    assert sonic.PAPER_T_TRANSMIT == (2.05, 4.1)
    assert 4.1 / 2.0 == pytest.approx(sonic.PAPER_T_TRANSMIT[0])


def test_break_even_near_the_measured_68_to_1():
    """The paper finds saturation at 270 processes on 4 GPUs (about 68 per GPU) with
    large batches; the model's t_ideal / t_gpu with its inputs is in that range."""
    lo = sonic.cpu_per_gpu(sonic.paper_job(link_gbps=2.0))
    hi = sonic.cpu_per_gpu(sonic.paper_job(link_gbps=1.0))
    assert 60 < lo < hi < 80
    assert lo <= 270 / 4 * 1.1


def test_unsaturated_time_is_flat_and_equals_t_ideal():
    job = sonic.paper_job()
    r = sonic.cpu_per_gpu(job)
    for n_cpu in (1, 10, 0.5 * r, 0.99 * r):
        assert not sonic.saturated(job, n_cpu, 1)
        assert sonic.t_sonic(job, n_cpu, 1) == pytest.approx(sonic.t_ideal(job))


def test_saturated_time_reduces_to_eq5_and_is_continuous():
    job = sonic.paper_job(dynamic_batching=False, large_batch=False)
    r = sonic.cpu_per_gpu(job)
    for n_cpu in (1.01 * r, 2 * r, 400):
        assert sonic.saturated(job, n_cpu, 1)
        assert sonic.t_sonic(job, n_cpu, 1) == pytest.approx(job.t_gpu * n_cpu)  # Eq. 5
    # continuous at the threshold, slope t_gpu / n_gpu after it
    assert sonic.t_sonic(job, r, 1) == pytest.approx(sonic.t_ideal(job))
    assert sonic.t_sonic(job, 4 * (r + 10), 4) - sonic.t_sonic(job, 4 * r, 4) == pytest.approx(job.t_gpu * 10)


def test_gb300_job_uses_the_measured_rate():
    job = sonic.gb300_job(hits_per_s=55_000 / 0.002)
    assert job.t_gpu == pytest.approx(0.002)
    assert job.t_latency == 0
    assert sonic.cpu_per_gpu(job) == pytest.approx((0.35 * 330 + 0.002) / 0.002)
    assert math.isfinite(sonic.t_sonic(job, 1e6, 1))
