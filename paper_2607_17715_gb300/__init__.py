"""GB300-native (sm_103a) C2KV compressed, composable KV-cache reuse: compose stored
per-chunk compressed KV into one GQA cache with RoPE re-rotation, then run the suffix
tokens' attention over it.  The compute lives in libc2kv.so (include/c2kv.h); the
Python module ``c2kv`` is its thin binding."""

__all__ = ["c2kv", "build"]
