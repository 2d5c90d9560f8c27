"""Algorithm 1 (Sec. 4.3) on hand cases, and FCFS against it in the simulator (CPU)."""
from paper_2601_11652_gb300 import scheduler as sch

# T_hat(B) = 1 ms per request + 1 us per cached token + 0.2 ms, in seconds
T = sch.BatchTime([1e-3, 0.0, 1e-6, 2e-4])


def _req(rid, arrival, k=4, ctx=1000, alpha=0.5, speed=4.0, t_draft=0.1, t_net=0.0):
    return sch.Request(rid, rid, arrival, k, ctx, alpha, speed, t_draft, t_net)


def test_request_estimates_follow_the_paper():
    r = _req(0, 10.0, k=4, alpha=0.5, speed=4.0, t_draft=0.1, t_net=0.05)
    assert r.gain == 2.0                                  # alpha * N_d
    assert abs(r.deadline - (10.0 + 2.0 / 4.0 - 0.15)) < 1e-12
    assert r.pages == (1000 + 5 + 15) // 16


def test_critical_requests_go_first_in_deadline_order():
    # r0 and r1 are critical at t (latest start passed), r1 has the earlier deadline; r2 is not
    reqs = [_req(0, 0.0, t_draft=0.09), _req(1, 0.0, t_draft=0.095), _req(2, 0.0, t_draft=-1.0)]
    # deadlines 0.41 and 0.405, solo cost T({i}) = 5 ms + 1 ms + 0.2 ms = 6.2 ms, delta 20 ms: both
    # latest starts (about 0.384 and 0.379) have passed at t = 0.39, and both fit:
    # t + T(two requests) = 0.39 + 0.0122 <= 0.405
    t = 0.39
    batch = sch.schedule_epoch(reqs, t, mem_budget=10**6, delta=0.02, T=T)
    assert [r.rid for r in batch][:2] == [1, 0]


def test_utility_order_and_stop_at_first_violation():
    # nobody is critical; higher alpha -> higher utility; a tight deadline stops the fill
    reqs = [_req(0, 0.0, alpha=0.2, t_draft=-1.0), _req(1, 0.0, alpha=0.9, t_draft=-1.0),
            _req(2, 0.0, alpha=0.6, t_draft=-1.0)]
    batch = sch.schedule_epoch(reqs, 0.0, mem_budget=10**6, delta=0.0, T=T)
    assert [r.rid for r in batch] == [1, 2, 0]
    # memory budget for two requests only: the lowest-utility one stays pending
    batch = sch.schedule_epoch(reqs, 0.0, mem_budget=2 * reqs[0].pages, delta=0.0, T=T)
    assert [r.rid for r in batch] == [1, 2]


def test_fcfs_takes_arrival_order():
    reqs = [_req(0, 2.0), _req(1, 1.0), _req(2, 3.0)]
    assert [r.rid for r in sch.schedule_fcfs(reqs, 5.0, 10**6, 2)] == [1, 0]


def test_slo_aware_scheduling_reduces_violations_under_load():
    # the batch time of this library's step (fitted on GB300, per cached token dominated), scaled
    # 40x to stand for a whole model's verification rather than one attention layer
    Tm = sch.BatchTime([40 * 1.27e-7, 0.0, 40 * 9.88e-10, 40 * 1.15e-4])
    fcfs = sch.simulate("fcfs", 200, Tm, horizon=20.0, seed=1, max_batch=32)
    wisp = sch.simulate("wisp", 200, Tm, horizon=20.0, seed=1)
    assert wisp.requests > 0 and fcfs.requests > 0
    assert wisp.violation_rate <= fcfs.violation_rate
