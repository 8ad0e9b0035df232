// wq4_host.h -- host-side helpers shared by the library's translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

namespace wq4 {

struct DeviceInfo {
    int sm_count = 0;
    int smem_optin = 0;      // max dynamic shared memory per block (opt-in)
    int coop_launch = 0;     // cooperative launch supported
};

// Properties of the current device, queried once per device.
const DeviceInfo* current_device_info(int* device_out);

// Device address of the library's status word on the current device.
uint32_t* status_word();

// 2-D tiled tensor map (driver entry point, no libcuda link): dims
// {inner, outer} elements, row pitch row_bytes, box {box_inner, box_outer}.
bool encode_tensor_map_2d(CUtensorMap* m, CUtensorMapDataType dt, const void* base, uint64_t inner,
                          uint64_t outer, uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer,
                          CUtensorMapSwizzle swz);

inline bool aligned(const void* p, size_t a)
{
    return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}

inline bool overlaps(const void* a, size_t na, const void* b, size_t nb)
{
    const uintptr_t pa = reinterpret_cast<uintptr_t>(a), pb = reinterpret_cast<uintptr_t>(b);
    return pa < pb + nb && pb < pa + na;
}

inline size_t align_up(size_t v, size_t a)
{
    return (v + a - 1) / a * a;
}

}  // namespace wq4
