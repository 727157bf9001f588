"""Layout helpers for the tests (token <-> image), independent of both sides."""
import numpy as np


def tokens_to_image(tok: np.ndarray, gh: int, gw: int) -> np.ndarray:
    """[B, gh*gw, C*4] tokens (c, ph, pw) -> [B, C, 2gh, 2gw] pixel image."""
    B, M, T = tok.shape
    C = T // 4
    t = tok.reshape(B, gh, gw, C, 2, 2)            # b y x c ph pw
    return t.transpose(0, 3, 1, 4, 2, 5).reshape(B, C, 2 * gh, 2 * gw)


def image_to_tokens(img: np.ndarray) -> np.ndarray:
    """[B, C, 2gh, 2gw] pixel image -> [B, gh*gw, C*4] tokens."""
    B, C, H2, W2 = img.shape
    gh, gw = H2 // 2, W2 // 2
    t = img.reshape(B, C, gh, 2, gw, 2).transpose(0, 2, 4, 1, 3, 5)
    return t.reshape(B, gh * gw, C * 4)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32)


def as_f32(a: np.ndarray) -> np.ndarray:
    return bf16_to_f32(a) if a.dtype == np.uint16 else np.asarray(a, np.float32)
