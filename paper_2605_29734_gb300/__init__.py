"""GB300-native hierarchical transition-attended memory lookup (HTAM, arxiv 2605.29734)."""
