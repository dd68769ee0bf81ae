"""Small test-side conversions between torch tensors and numpy arrays."""
import numpy as np
import torch


def np_bytes(t: torch.Tensor) -> np.ndarray:
    """The raw bytes of a tensor (copied to the host) as uint8."""
    t = t.detach().contiguous().cpu()
    if t.dtype == torch.bfloat16:
        t = t.view(torch.int16)
    return t.numpy().view(np.uint8).reshape(-1)


def np_view(t: torch.Tensor) -> np.ndarray:
    """Host numpy array of a tensor; bfloat16 is carried as uint16 bits."""
    t = t.detach().contiguous().cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def u64(t: torch.Tensor) -> list:
    return [int(x) for x in t.detach().cpu().numpy().view(np.uint64)]
