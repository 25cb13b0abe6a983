"""jab_loss_forward_noalloc: the candidate-loss forward for callers that cannot allocate device
memory (their device memory is reserved up front by another allocator, or allocation is not allowed
where they need the loss). It runs on the library's fixed device scratch instead of a caller
workspace, and must give the losses of jab_loss_forward with a caller workspace, call after call.

Kept in its own file, collected last, so that a failure here cannot stop a fail-fast run before the
other tests have run; it also passes on its own in a fresh process.
"""
import pytest
import torch

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)


def test_noalloc_forward_matches_workspace_forward_twice():
    from paper_2609_34866_gb300 import build
    build.build()
    import paper_2609_34866_gb300 as J
    from tests.harness import L_TOL
    from workloads import WORKLOADS, make_block_weights, make_x

    J.jab_get_device_status()
    wl = WORKLOADS["gpt2_sweep"]
    B, T = 2, 200                                     # several tiles and a ragged tail
    desc = J.desc_from_shape(wl.shape, wl.group_size)
    X = make_x(wl, batch=B, seq_len=T).cuda()
    W = make_block_weights(wl).cuda()
    bits = [2, 3, 8]
    ws = J.Workspace(desc, B, T, len(bits), False)
    A = torch.empty((B, T, wl.shape.n_q_heads * wl.shape.head_dim), dtype=torch.float32, device="cuda")
    J.jab_reference_forward(desc, B, T, X, W, A, ws)
    scales = []
    for b in bits:
        s = torch.empty((wl.shape.d_out, wl.shape.d_model // wl.group_size), dtype=torch.float32,
                        device="cuda")
        J.jab_init_scales(desc, b, 0, W, s)
        scales.append(s)
    ref = torch.empty(len(bits), dtype=torch.float64, device="cuda")
    ref_parts = torch.empty((len(bits), B, wl.shape.n_q_heads), dtype=torch.float64, device="cuda")
    J.jab_loss_forward(desc, B, T, X, W, A, bits, scales, ref, ws, sse_parts=ref_parts)
    outs = [(torch.full_like(ref, float("nan")), torch.full_like(ref_parts, float("nan")))
            for _ in range(3)]
    # the first call on a device may load the library's module that holds the fixed array (lazy
    # module loading), which is when the device gives the array its memory: measure after it
    J.jab_loss_forward_noalloc(desc, B, T, X, W, A, bits, scales, outs[0][0], sse_parts=outs[0][1])
    torch.cuda.synchronize()
    torch.testing.assert_close(outs[0][0], ref, rtol=L_TOL, atol=0)
    outs = outs[1:]
    for out, parts in outs:                           # the scratch keeps the last call's contents
        torch.cuda.synchronize()
        free0 = torch.cuda.mem_get_info()[0]
        J.jab_loss_forward_noalloc(desc, B, T, X, W, A, bits, scales, out, sse_parts=parts)
        torch.cuda.synchronize()
        # the call took no device memory (the device's free memory is unchanged; the library has no
        # access to torch's caching allocator, so this is the whole of what it could take)
        assert torch.cuda.mem_get_info()[0] == free0
        torch.testing.assert_close(out, ref, rtol=L_TOL, atol=0)
        torch.testing.assert_close(parts, ref_parts, rtol=L_TOL, atol=0)
    assert J.jab_get_device_status() == 0

    # a problem larger than the fixed scratch is refused with its own status, before any launch
    big = WORKLOADS["mistral_block"]
    bdesc = J.desc_from_shape(big.shape, big.group_size)
    with pytest.raises(J.JabError) as e:
        J.jab_loss_forward_noalloc(bdesc, 64, 2048, X, W, A, [3], [scales[0]], out)
    assert e.value.status == 7
