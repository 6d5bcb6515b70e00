"""GB300-native Distance-KV inference hot path (pattern map, prune-and-pack,
split-K decode attention) behind the C ABI of include/dkv.h."""
