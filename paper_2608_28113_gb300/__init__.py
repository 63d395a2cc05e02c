"""GB300-native H-Scale hot path (placeholder; the binding is added with the CUDA library)."""
