"""GB300-native activation-sparse dReLU FFN (Turbo Sparse, arXiv 2406.05955)."""
