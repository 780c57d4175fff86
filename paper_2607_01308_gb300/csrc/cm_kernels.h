// Internal interface between the host core (cm_host.cpp) and the CUDA kernels: the
// content-address kernels (cm_hash_kernels.h), the render kernel (cm_render_kernels.h)
// the byte comparison of the re-delivery fast path (cm_dedup_kernels.h) and the readback
// of small results (cm_readback_kernels.h). Not part of the public ABI.
#pragma once

#include "cm_dedup_kernels.h"
#include "cm_hash_kernels.h"
#include "cm_readback_kernels.h"
#include "cm_render_kernels.h"
