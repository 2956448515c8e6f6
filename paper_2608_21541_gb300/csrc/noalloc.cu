// noalloc.cu — decode attention that allocates nothing.
//
// certkv_decode_attn needs a caller-provided scratch buffer for its split-K
// partial results.  Some callers cannot provide one: a plugin that an
// inference server hands only its input and output tensors, or a per-token
// decode loop that must not call cudaMalloc because cudaMalloc can wait for
// the whole device and breaks a memory plan fixed at start-up.  This entry
// point runs the same decode kernels with their scratch in a fixed-size array
// that lives in the library's own device memory, reserved when the library is
// loaded and kept until the process exits.
#include <mutex>

#include "../../include/certkv.h"
#include "internal.cuh"

namespace certkv {

// The scratch shared by every call on a device.  Its size is the public limit
// CERTKV_NOALLOC_SCRATCH_BYTES.
static __device__ __align__(256) unsigned char g_noalloc_scratch[CERTKV_NOALLOC_SCRATCH_BYTES];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};
}  // namespace

}  // namespace certkv

extern "C" int certkv_decode_attn_noalloc(const certkv_shape* shape, const void* q,
                                          const certkv_packed* packed, float scale,
                                          int32_t tail_slot, void* out, void* stream) {
  using namespace certkv;
  // The same validation as certkv_decode_attn, with the size limit checked
  // right after the shape: a call that is too large is refused before its
  // pointers are looked at.
  Prob p;
  int rc = decode_prob(shape, &p);
  if (rc) return rc;
  if (decode_workspace(p) > (size_t)CERTKV_NOALLOC_SCRATCH_BYTES) return CERTKV_ETOOLARGE;
  float sc = 0.0f;
  if ((rc = decode_args(shape, q, packed, scale, tail_slot, out, &sc))) return rc;
  p.capacity = packed->capacity_slots;

  // Set-up, once per device and with that device current: the device address
  // of the static scratch array.
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return CERTKV_ECUDA;
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> g(g_mu);
    if (!g_scratch_ptr[dev]) {
      void* ptr = nullptr;
      if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || !ptr) return CERTKV_ECUDA;
      g_scratch_ptr[dev] = ptr;
    }
    scratch = g_scratch_ptr[dev];
  }
  if (!launch_decode(p, q, packed->k, packed->v, packed->offsets, packed->real_counts, tail_slot,
                     sc, out, reinterpret_cast<char*>(scratch),
                     reinterpret_cast<cudaStream_t>(stream)))
    return CERTKV_ECUDA;
  return cudaGetLastError() == cudaSuccess ? CERTKV_OK : CERTKV_ECUDA;
}
