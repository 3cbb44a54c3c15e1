"""The device-side timeout path, exercised on the GPU without a fault or a
hang.

Every wait in the kernels gives up after the library's wait limit, sets the
timeout bit of the workspace status word and lets its kernel return, so that
mcpu_read_device_status reports MCPU_ERR_TIMEOUT and the CUDA context stays
usable. No input can make one of those waits run out, so
mcpu_selftest_wait_timeout builds the situation itself: a warp waits, with
the decode kernels' own bounded wait, on a barrier that nothing completes.
The test checks that the wait ends after (and not long after) its limit, that
the status reaches the host, and that the same workspace, once reset, serves
a normal append + forward that matches the oracle.
"""
import numpy as np
import pytest
import torch

import workloads as W

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from _gpu import Run, assert_parity, oracle_full
    from paper_2608_22167_gb300 import mcpu


def test_wait_gives_up_reports_timeout_and_leaves_the_context_usable():
    batch = W.config_tiny()
    run = Run(batch)
    mcpu.mcpu_reset_device_status(run.ws)
    report = torch.full((4,), -1, dtype=torch.int64, device="cuda")
    mcpu.mcpu_selftest_wait_timeout(run.ws, report)
    code, bits = run.status()  # synchronises the stream
    done_ok, never_ok, waited_ns, limit_ns = (int(x) for x in report.cpu())
    assert done_ok == 1, "a wait whose phase completed did not return success"
    assert never_ok == 0, "a wait on a barrier that nothing completes returned success"
    assert limit_ns > 0
    assert limit_ns <= waited_ns < 20 * limit_ns, (waited_ns, limit_ns)
    assert code == 7 and bits & mcpu.STATUS_TIMEOUT, (code, bits)

    # the context survived: the same workspace, reset, serves a normal call
    mcpu.mcpu_reset_device_status(run.ws)
    run.append()
    run.forward()
    code, bits = run.status()
    assert code == 0, f"device status bits {bits}"
    ref_out, ref_lse, (okc, ovc) = oracle_full(batch)
    assert np.array_equal(W.to_host(run.kc), okc), "k pool differs after append"
    assert np.array_equal(W.to_host(run.vc), ovc), "v pool differs after append"
    got_out, got_lse = run.out_host()
    assert_parity(got_out, got_lse, ref_out, ref_lse, "tiny batch after the timeout check")


@pytest.mark.parametrize("role", [0, 1, 2], ids=["softmax", "producer", "issuer"])
def test_append_kernel_abort_reaches_every_role(role):
    # The tcgen05 append kernel's own waits, in its self-test form: one role
    # (softmax warps of tile A, the TMA producer, or tile A's MMA issuer)
    # stops at the second key block of its first item and waits on a barrier
    # nothing completes for half the wait limit, then raises the CTA's abort
    # flag. Every other role is then blocked on that role and waits with the
    # full limit: each must leave on the flag (the flag keeps the stalled
    # role's mark, nobody left at the full limit), the issuers and the
    # producer drain what they had in flight, TMEM is freed, the timeout bit
    # reaches the host, and the next normal call on every SM matches the oracle.
    batch = W.build_batch("abort", 91 + role, [300, 40, 700], [300, 1, 90], 16, 2)
    run = Run(batch)
    run.append()
    mcpu.mcpu_reset_device_status(run.ws)
    report = torch.full((16,), -1, dtype=torch.int64, device="cuda")
    mcpu.mcpu_selftest_append_abort(run.q, run.kc, run.vc, run.bt, run.sl, run.qsl, batch.softmax_scale, run.out,
                                    run.lse, run.ws, role, report)
    code, bits = run.status()  # synchronises the stream
    r = [int(x) for x in report.cpu()]
    flag, exits, stall_ns, limit_ns, freed = r[0], r[1:12], r[12], r[13], r[14]
    assert code == 7 and bits & mcpu.STATUS_TIMEOUT, (code, bits)
    assert flag == 2, f"a role ran out of its own wait instead of leaving on the abort flag: {r}"
    assert freed == 1, "TMEM was not freed"
    assert 0 < stall_ns < limit_ns
    # every warp left after the stall ended and well before its own limit
    for w, e in enumerate(exits):
        assert stall_ns <= e < stall_ns + (limit_ns - stall_ns) // 2, (w, e, stall_ns, limit_ns)

    # TMEM and the context are intact: a normal call (one append CTA per SM)
    mcpu.mcpu_reset_device_status(run.ws)
    run.forward()
    code, bits = run.status()
    assert code == 0, f"device status bits {bits}"
    ref_out, ref_lse, _ = oracle_full(batch)
    got_out, got_lse = run.out_host()
    assert_parity(got_out, got_lse, ref_out, ref_lse, f"batch after the abort check (role {role})")
