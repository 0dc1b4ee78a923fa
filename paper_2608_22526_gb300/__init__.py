"""RS3-Prune hot path on GB300: CUDA library librs3 (include/rs3.h) and its binding."""
