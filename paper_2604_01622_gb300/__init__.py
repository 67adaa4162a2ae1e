"""GB300-native expert-choice MoE layer (placeholder; binding added with the library)."""
