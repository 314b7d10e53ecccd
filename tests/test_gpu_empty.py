"""Empty batches through the binding on the GPU: zero rows or groups is a
valid call that launches nothing and leaves every buffer as it was."""
import pytest

from paper_2607_20791_gb300 import binding

pytestmark = pytest.mark.gpu


def test_empty_batches_through_the_binding(gpu_lib):
    import torch
    dev = "cuda"
    i32, u8, f32 = torch.int32, torch.uint8, torch.float32
    # sample head with no rows
    binding.rgd_sample_head(torch.empty(0, 128, device=dev), None, torch.empty(0, device=dev),
                            torch.empty(0, device=dev), torch.empty(0, dtype=torch.int64, device=dev), 0, None,
                            torch.empty(0, dtype=i32, device=dev))
    # gate calls with no groups
    trie = binding.Trie([[1, 2], [1, 3, 4]], 2)
    st = binding.new_gate_state(0)
    binding.rgd_gate_state_init(st, 0)
    binding.rgd_probe_gate(trie, 0, 2, torch.empty(0, dtype=i32, device=dev), 1, 1, -1, 8, st)
    tok = torch.full((1,), 7, dtype=i32, device=dev)
    binding.rgd_soft_gate(trie, 0, 2, torch.empty(0, 16, device=dev), 32, 4, 0.1, 2, -1, 8, st, tok)
    binding.rgd_residual_precheck(torch.empty(0, 64, device=dev), torch.zeros(64, dtype=f32, device=dev), 0.0, 0.5,
                                  2, st)
    # a step with no probe tokens leaves the states alone
    st1 = binding.new_gate_state(3)
    binding.rgd_gate_state_init(st1, 3)
    before = st1.clone()
    binding.rgd_probe_gate(trie, 3, 2, torch.zeros(3, dtype=i32, device=dev), 0, 1, -1, 8, st1,
                           torch.ones(6, dtype=u8, device=dev))
    torch.cuda.synchronize()
    assert torch.equal(st1, before) and int(tok.item()) == 7
    trie.close()
