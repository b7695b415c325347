"""Pins for the chained step's attention link (oracle.attention_link, CPU): attention of the new
tokens over a KV cache between QKV and O.  Each case has a result fixed without the oracle's own
formula: an empty cache and one token reduce to the one-position V slice the plain chain uses; a
new token never sees a later one; the cache holds exactly the new tokens' k and v afterwards; keys
that are all zero give the plain average of the values."""
import numpy as np

import oracle
import synth

D = 128


def qkv(M, n_heads, seed, scale=1.0):
    H = n_heads * D
    b = synth.normal_bf16(synth.key(seed, 7), 1.0, M * 3 * H).reshape(M, 3 * H)
    return ((b.astype(np.uint32) << 16).view(np.float32) * np.float32(scale)).astype(np.float32)


def cache(n_heads, L_max, seed):
    return synth.normal_bf16(synth.key(seed, 8), 1.0, 2 * n_heads * L_max * D).reshape(2, n_heads, L_max, D)


def test_empty_cache_single_token_is_the_v_slice():
    n_heads = 4
    y = qkv(1, n_heads, 1)
    x, kv = oracle.attention_link(y, cache(n_heads, 8, 1), 0, n_heads)
    H = n_heads * D
    assert np.array_equal(x, oracle.slice_x(y, 2 * H, H))


def test_cache_receives_the_new_tokens_and_nothing_else():
    n_heads, L_max, L_past, M = 3, 40, 17, 3
    y = qkv(M, n_heads, 2)
    kv0 = cache(n_heads, L_max, 2)
    _, kv = oracle.attention_link(y, kv0, L_past, n_heads)
    H = n_heads * D
    k_new = oracle.slice_x(y, H, H).reshape(M, n_heads, D).transpose(1, 0, 2)
    v_new = oracle.slice_x(y, 2 * H, H).reshape(M, n_heads, D).transpose(1, 0, 2)
    assert np.array_equal(kv[0, :, L_past:L_past + M], k_new)
    assert np.array_equal(kv[1, :, L_past:L_past + M], v_new)
    keep = np.ones(L_max, bool)
    keep[L_past:L_past + M] = False
    assert np.array_equal(kv[:, :, keep], kv0[:, :, keep])
    assert np.array_equal(kv0, cache(n_heads, L_max, 2)), "the input cache was modified"


def test_new_tokens_are_causal():
    n_heads, L_past, M = 2, 5, 3
    H = n_heads * D
    y = qkv(M, n_heads, 3)
    kv = cache(n_heads, 16, 3)
    x, _ = oracle.attention_link(y, kv, L_past, n_heads)
    y2 = y.copy()
    y2[2, H:] = -y2[2, H:]            # the last token's k and v
    x2, _ = oracle.attention_link(y2, kv, L_past, n_heads)
    assert np.array_equal(x[:2], x2[:2]) and not np.array_equal(x[2], x2[2])
    y3 = y.copy()
    y3[1, H:] *= 2                    # the middle token's k and v
    x3, _ = oracle.attention_link(y3, kv, L_past, n_heads)
    assert np.array_equal(x[0], x3[0]) and not np.array_equal(x[1], x3[1])


def test_zero_keys_average_the_values():
    """Zero keys give every visible position the same score, so out is the mean of the visible
    values: with small-integer values and four positions the mean is exact in bf16."""
    n_heads, L_past, M = 2, 3, 1
    H = n_heads * D
    y = qkv(M, n_heads, 4)
    y[:, H:2 * H] = 0.0                                        # the new token's key
    vals = np.arange(4 * n_heads * D).reshape(4, n_heads, D) % 7 - 3.0   # exact in bf16
    kv = np.zeros((2, n_heads, 8, D), np.uint16)
    kv[1, :, :L_past] = (vals[:L_past].transpose(1, 0, 2).astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    y[0, 2 * H:] = vals[L_past].reshape(-1)
    x, _ = oracle.attention_link(y, kv, L_past, n_heads)
    mean = vals.mean(axis=0).reshape(-1)                       # multiples of 1/4, |mean| <= 3
    assert np.array_equal(x[0], (mean.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16))
