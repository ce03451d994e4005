"""GB300-native (sm_103a) homogenized StackLSTM step, forward and backward.

The hot path of Ding & Koehn, "Parallelizable Stack Long Short-Term Memory": every
instance of a minibatch runs the same step whatever its stack op (Algorithm 1), so the
whole batch is one gate contraction per step. The kernels live in ``csrc/`` and are
reached through the C ABI of ``include/stacklstm.h``; ``binding`` is its thin Python
binding, ``runner`` moves synthetic workloads to and from the device, ``workloads``
draws them.
"""
from .binding import (SL_BF16, SL_FP32, StackLSTMError, StackLSTMHandle, load, stacklstm_backward,
                      stacklstm_create, stacklstm_destroy, stacklstm_forward, stacklstm_set_async,
                      stacklstm_get_timing, stacklstm_pointers_noalloc, stacklstm_set_stream, stacklstm_set_timing, stacklstm_status,
                      stacklstm_status_string)

__all__ = ["SL_BF16", "SL_FP32", "StackLSTMError", "StackLSTMHandle", "load", "stacklstm_backward",
           "stacklstm_create", "stacklstm_destroy", "stacklstm_forward", "stacklstm_set_async",
           "stacklstm_get_timing", "stacklstm_pointers_noalloc", "stacklstm_set_stream", "stacklstm_set_timing", "stacklstm_status",
           "stacklstm_status_string"]
