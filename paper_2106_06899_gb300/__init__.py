"""Top-k attention (arxiv 2106.06899) on GB300: C-ABI CUDA library + thin Python binding."""
