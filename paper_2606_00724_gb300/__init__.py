"""WaveFilter hot path for GB300 (sm_103a): Haar-DWT KV filtering and sparse attention."""
