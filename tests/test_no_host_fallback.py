"""The Python binding marshals device pointers only: host tensors are refused
before anything reaches the library, so there is no CPU path to fall into --
CPU only (no compute calls)."""
import pytest
import torch


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    __graft_entry__._load_builder().build()
    import paper_2510_16292_gb300 as q
    return q


def test_host_tensors_are_refused(lib):
    i32 = torch.zeros(4, dtype=torch.int32)
    bf = torch.zeros((64, 256), dtype=torch.bfloat16)
    O = torch.zeros((4, 256), dtype=torch.float32)
    cache = lib.LatentCache(torch.zeros((1, 8, 64), dtype=torch.int8), torch.zeros((1, 8), dtype=torch.float32),
                            8, 1, 8, 64)
    calls = [
        lambda: lib.qsvd_quantize_weight(torch.zeros((256, 64), dtype=torch.float32)),
        lambda: lib.qsvd_quantize_weight(torch.zeros((256, 64), dtype=torch.float32), rot=256),
        lambda: lib.qsvd_latent_decode_attn(cache, i32, 4, bf, bf, bf, 2, 128, O, workspace=torch.zeros(16, dtype=torch.uint8)),
        lambda: lib.qsvd_latent_prefill_attn(cache, i32, i32, 4, bf, bf, bf, 2, 128, O,
                                             workspace=torch.zeros(16, dtype=torch.uint8)),
        lambda: lib.qsvd_prefill_weights(bf, bf, bf),
        lambda: lib.qsvd_latent_prefill(cache, [(0, 0, 4)], torch.zeros((768, 64), dtype=torch.float16), 2, 128, O,
                                        workspace=torch.zeros(16, dtype=torch.uint8)),
        lambda: lib.qsvd_decode_step(lib.DownWeight(torch.zeros((64, 256), dtype=torch.int8),
                                                    torch.zeros((64, 256), dtype=torch.bfloat16),
                                                    torch.zeros(64, dtype=torch.float32)),
                                     bf[:1], cache, i32[:1], 4, bf, bf, bf, 2, 128, O[:1],
                                     workspace=torch.zeros(16, dtype=torch.uint8)),
        lambda: lib.qsvd_beta_factors(torch.zeros((64, 32), dtype=torch.float64),
                                      torch.zeros((32, 128), dtype=torch.float64),
                                      torch.ones(32, dtype=torch.float64), torch.ones(32, dtype=torch.float64)),
        lambda: lib.qsvd_beta_objective(torch.zeros((4, 128), dtype=torch.float32), torch.zeros((4, 32), dtype=torch.int8),
                                        torch.zeros(4, dtype=torch.float32), 8, 32,
                                        lib.UpWeight(torch.zeros((32, 128), dtype=torch.int8),
                                                     torch.zeros(128, dtype=torch.float32), 8),
                                        workspace=torch.zeros(16, dtype=torch.uint8)),
    ]
    for call in calls:
        with pytest.raises(ValueError, match="device tensor expected"):
            call()
