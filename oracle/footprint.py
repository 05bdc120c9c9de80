"""KV cache footprint, Eq. 1 (Sec. 4.1): D_KV = 2 * L * n_kv * d_h * s_ctx * b.

TEST INFRASTRUCTURE ONLY (see the package docstring).

The factor 2 counts K and V; b is bytes per element (2 for FP16 / bf16).  With
paging, whole pages of P tokens are held, so the bytes a paged cache holds for
a sequence of n tokens are Eq. 1 evaluated at s_ctx = P * ceil(n / P).
"""


def kv_bytes_eq1(L: int, n_kv: int, d_h: int, s_ctx: int, b: int = 2) -> int:
    """Eq. 1 for one request of s_ctx cached tokens."""
    return 2 * L * n_kv * d_h * s_ctx * b


def kv_bytes_paged(L: int, n_kv: int, d_h: int, P: int, lens, b: int = 2) -> int:
    """Bytes held by a paged cache for sequences of the given token counts."""
    return sum(kv_bytes_eq1(L, n_kv, d_h, P * ((int(n) + P - 1) // P), b) for n in lens)
