"""GB300-native (sm_103a) KV-cache splicing hot path of Nexus.

``nexus``      ctypes binding of the C-ABI library ``libnexus.so``
``workloads``  seeded synthetic inputs shaped like Qwen2.5-14B attention
"""
