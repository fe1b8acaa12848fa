"""GB300-native QuantWM per-chunk 2-bit KV-cache path (placeholder, filled in below)."""
