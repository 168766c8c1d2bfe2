"""GB300-native TGV-KV eviction (placeholder; binding added with the library)."""
