// status.cuh -- the device status word the kernels report into.
#pragma once
#include <cuda_runtime.h>

namespace rdn {
// Device address, on the current device, of the library's status word: a
// kernel whose bounded wait gives up (or whose shared memory is misaligned)
// stores RDN_ERR_TIMEOUT / RDN_ERR_CUDA there and skips the rest of its work;
// rdn_device_status() reads and clears it.  NULL if the lookup failed (the
// kernels then report nothing).  Defined in api.cu.
int *status_word();

// Host-side fault injection for tests, from the environment variable
// RDN_FAULT_INJECT read at each call: "workspace" (1) makes the forward and
// backward entry points fail their workspace check, "launch" (2) makes them
// fail as a launch would, both after argument validation and before
// anything is enqueued; "device_wait" (3) makes the tensor-core forward scan
// skip one MMA completion signal, so that its bounded wait gives up
// (RDN_ERR_TIMEOUT in the status word) and the kernel drains and exits;
// "device_wait_bwd" (4) does the same in the tensor-core backward chain.
// 0 when unset or unrecognised.  Defined in api.cu.
int fault_injection();
}  // namespace rdn
