"""GB300-native (sm_103a) C-ABI library for the ReCo hot path.

ReCo ("Fewer Tokens, Smaller Cache: Reward-Coordinated Efficient Reasoning")
compresses a reasoning model's KV cache at every step boundary: a process reward
sets a retention ratio (Eq. 1), cached tokens are scored by the attention they get
from a window of recent queries (Eq. 2), the best tokens per KV head are kept and
compacted in place, and decode attention runs over the ragged compacted cache.
A reward-banded penalty on reflection-token logits (Eq. 3-4) and the answer-
perplexity stop test (Eq. 5-6) run alongside.

``reco`` is the thin ctypes binding over ``libreco.so`` (names match the C ABI in
include/reco.h); ``workloads`` holds the seeded synthetic input generators.
Importing this package loads nothing; the first call into ``reco`` loads the
library and raises if it has not been built.
"""
