// tcgen05 / TMEM gather-decode (sm_103a).
#include "ntc_internal.cuh"

namespace ntc {

size_t tc_image_bytes(uint32_t H) { return (size_t)H * 16; }

}  // namespace ntc
