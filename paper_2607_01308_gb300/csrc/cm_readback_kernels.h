// Internal interface between the host core (cm_host.cpp) and the readback kernel
// (readback.cu). Not part of the public ABI.
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

namespace cm {

// Copies `bytes` (a multiple of 4, both addresses 4-byte aligned) from device memory to
// pinned host memory through its device-mapped address, with the SMs' stores over the
// host link instead of a copy engine: a small result read this way does not queue
// behind bulk device-to-host copies that other streams have in flight.
cudaError_t launch_readback(void *host_mapped_dst, const void *src, size_t bytes,
                            cudaStream_t stream);

}  // namespace cm
