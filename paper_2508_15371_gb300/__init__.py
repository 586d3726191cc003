"""GB300-native CM-ASD logits pass (arXiv 2508.15371): confidence signals,
next draft length, confidence-modulated acceptance, first-reject scan and
correction token, behind the C-ABI library libcmsd.so."""
