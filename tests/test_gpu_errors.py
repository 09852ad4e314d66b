"""Error behaviour of the C ABI: host-side checks reject bad calls before any launch
(SPEC_EINVAL / SPEC_ESTATE, state unchanged), and data-dependent faults found by the kernels'
own bounds checks set the device guard flag, reported by spec_sync as SPEC_EDEVICE, without
trapping: the context stays usable afterwards."""
import pytest
import torch

import synth_inputs as S
from paper_2609_03181_gb300 import fastmtp as F

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def eng():
    shape = S.ModelShape(n_layers=1, vocab=1024)
    vw = S.verifier_weights(shape, 9)
    dw = S.draft_weights(shape, 9)
    e = F.Engine(vw, dw, max_batch=2, K_max=3, max_ctx=200, page_size=64)
    for b in range(2):
        e.load_prefix(b, S.kv_prefix(9, b, 1, 50, 10, 128), S.draft_kv_prefix(9, b, 50, 10, 128), 7)
    yield e
    e.close()


def _bufs(B, K):
    dev = torch.device("cuda")
    return (torch.arange(B, dtype=torch.int32, device=dev), torch.empty(B, K + 1, dtype=torch.int32, device=dev),
            torch.empty(B, dtype=torch.int32, device=dev))


def test_host_side_rejections(eng):
    slots, vt, acc = _bufs(2, 3)
    cand = torch.tensor([[7, 1, 2, 3]] * 2, dtype=torch.int32, device="cuda")
    big = torch.arange(3, dtype=torch.int32, device="cuda")
    with pytest.raises(F.FastMTPError) as e:
        eng.verify_step(big, torch.zeros(3, 4, dtype=torch.int32, device="cuda"), vt, acc)   # B > max_batch
    assert e.value.status == F.SPEC_EINVAL
    with pytest.raises(F.FastMTPError) as e:
        eng.verify_step(slots, torch.zeros(2, 6, dtype=torch.int32, device="cuda"), vt, acc)  # K > K_max
    assert e.value.status == F.SPEC_EINVAL
    with pytest.raises(F.FastMTPError) as e:
        eng.accept_commit(slots, vt, acc)                                                        # nothing verified
    assert e.value.status == F.SPEC_ESTATE
    eng.draft_step(slots, 3, vt)           # passes the host checks; the slots have no queued rows
    with pytest.raises(F.FastMTPError) as e:
        eng.sync()
    assert e.value.status == F.SPEC_EDEVICE and "0x10" in str(e.value)
    eng.verify_step(slots, cand, vt, acc)
    with pytest.raises(F.FastMTPError) as e:
        eng.verify_step(slots, cand, vt, acc)                                                   # not committed yet
    assert e.value.status == F.SPEC_ESTATE
    com, nc = torch.empty(2, 4, dtype=torch.int32, device="cuda"), torch.empty(2, dtype=torch.int32, device="cuda")
    eng.accept_commit(slots, com, nc)
    eng.sync()


def test_device_guard_flags_and_recovery(eng):
    slots, vt, acc = _bufs(2, 1)
    for b in range(2):
        eng.load_prefix(b, S.kv_prefix(9, b, 1, 50, 10, 128), S.draft_kv_prefix(9, b, 50, 10, 128), 7)
    # token id outside the vocabulary
    eng.verify_step(slots, torch.tensor([[7, 5000], [7, 1]], dtype=torch.int32, device="cuda"), vt, acc)
    eng.accept_commit(slots, torch.empty(2, 2, dtype=torch.int32, device="cuda"), acc)
    with pytest.raises(F.FastMTPError) as e:
        eng.sync()
    assert e.value.status == F.SPEC_EDEVICE and "0x2" in str(e.value)
    # candidate 0 that is not the pending token
    for b in range(2):
        eng.load_prefix(b, S.kv_prefix(9, b, 1, 50, 10, 128), S.draft_kv_prefix(9, b, 50, 10, 128), 7)
    eng.verify_step(slots, torch.tensor([[8, 1], [7, 1]], dtype=torch.int32, device="cuda"), vt, acc)
    eng.accept_commit(slots, torch.empty(2, 2, dtype=torch.int32, device="cuda"), acc)
    with pytest.raises(F.FastMTPError) as e:
        eng.sync()
    assert "0x8" in str(e.value)
    # the context keeps working after the flag was reported
    for b in range(2):
        eng.load_prefix(b, S.kv_prefix(9, b, 1, 50, 10, 128), S.draft_kv_prefix(9, b, 50, 10, 128), 7)
    eng.verify_step(slots, torch.tensor([[7, 1], [7, 2]], dtype=torch.int32, device="cuda"), vt, acc)
    eng.accept_commit(slots, torch.empty(2, 2, dtype=torch.int32, device="cuda"), acc)
    eng.sync()
    assert eng.seq_state(0)[0] == 50 + int(acc[0])


def test_slot_id_out_of_range_sets_guard_flag(eng):
    """A slot id in the device slots array outside [0, max_batch) is caught by every kernel that
    indexes by slot: its sequence is skipped (no page, state or staging access) and the flag
    reads 64; the valid sequence of the same call is still committed."""
    dev = torch.device("cuda")
    for b in range(2):
        eng.load_prefix(b, S.kv_prefix(9, b, 1, 50, 10, 128), S.draft_kv_prefix(9, b, 50, 10, 128), 7)
    bad = torch.tensor([0, 1 << 20], dtype=torch.int32, device=dev)
    vt = torch.empty(2, 2, dtype=torch.int32, device=dev)
    acc = torch.empty(2, dtype=torch.int32, device=dev)
    eng.verify_step(bad, torch.tensor([[7, 1], [7, 2]], dtype=torch.int32, device=dev), vt, acc)
    eng.accept_commit(bad, torch.empty(2, 2, dtype=torch.int32, device=dev), acc)
    with pytest.raises(F.FastMTPError) as e:
        eng.sync()
    assert e.value.status == F.SPEC_EDEVICE and "0x40" in str(e.value)
    assert eng.seq_state(0)[0] == 50 + int(acc[0])
    assert eng.seq_state(1)[0] == 50
    # the draft head's kernels check the same ids
    eng.draft_step(bad, 1, torch.empty(2, 2, dtype=torch.int32, device=dev))
    with pytest.raises(F.FastMTPError) as e:
        eng.sync()
    assert "0x40" in str(e.value) or "0x50" in str(e.value)
