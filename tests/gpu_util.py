"""Helpers shared by the GPU tests: run poseidon_eval_batch on device
buffers through the C ABI."""
import numpy as np


def eval_device(P, handle, cands, stream=None):
    import torch
    n = len(cands)
    d_c = torch.from_numpy(np.ascontiguousarray(cands).view(np.uint8)).cuda()
    d_T = torch.full((max(n, 1),), -7, dtype=torch.int32, device="cuda")
    d_F = torch.full((max(n, 1),), 99, dtype=torch.uint8, device="cuda")
    s = stream if stream is not None else torch.cuda.current_stream()
    P.poseidon_eval_batch(handle, d_c.data_ptr(), n, d_T.data_ptr(), d_F.data_ptr(),
                          s.cuda_stream)
    torch.cuda.synchronize()
    return d_T[:n].cpu().numpy(), d_F[:n].cpu().numpy()


def eval_device_ex(P, handle, cands, stream=None):
    """poseidon_eval_batch_ex on 24-byte records (a TP index per stage)."""
    import torch
    n = len(cands)
    d_c = torch.from_numpy(np.ascontiguousarray(cands).view(np.uint8)).cuda()
    d_T = torch.full((max(n, 1),), -7, dtype=torch.int32, device="cuda")
    d_F = torch.full((max(n, 1),), 99, dtype=torch.uint8, device="cuda")
    s = stream if stream is not None else torch.cuda.current_stream()
    P.poseidon_eval_batch_ex(handle, d_c.data_ptr(), n, d_T.data_ptr(), d_F.data_ptr(),
                             s.cuda_stream)
    torch.cuda.synchronize()
    return d_T[:n].cpu().numpy(), d_F[:n].cpu().numpy()
