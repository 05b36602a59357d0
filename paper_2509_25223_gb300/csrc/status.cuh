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
}  // namespace rdn
