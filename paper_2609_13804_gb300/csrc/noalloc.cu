// sp_select_noalloc: sp_select for callers that cannot allocate device memory.
//
// Some callers have no way to obtain a device workspace: a plug-in living inside
// a host application that owns every byte of device memory through its own
// pool, a plain-C caller without any allocator of its own, or a latency-bound
// path that may not pay for cudaMalloc (which can synchronise the device).
// This entry point runs exactly the selection of sp_select, but its scratch is
// a file-scope __device__ array of fixed size instead of a caller workspace.
//
// Cost and limits:
//   * the array (SP_SELECT_NOALLOC_SCRATCH_BYTES) is part of the library's
//     device image, so every GPU on which the library is loaded holds it until
//     the process exits;
//   * a batch whose sp_select_workspace() exceeds it is rejected with
//     SP_ERR_WORKSPACE before anything is launched;
//   * every call shares the one array: calls whose GPU work overlaps (two
//     streams, two host threads) race on it; serialise them;
//   * the array's device address is looked up once per device and kept for
//     the life of the process: after cudaDeviceReset (or any other teardown of
//     the device's primary context) it is stale, so do not use this entry
//     point across a device reset.
#include <cuda_runtime.h>

#include <mutex>

#include "internal.h"

namespace {

constexpr size_t kScratchBytes = SP_SELECT_NOALLOC_SCRATCH_BYTES;

__device__ __align__(256) unsigned char g_select_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of g_select_scratch on the current device.  In host code the
// array's name is only a host-side stand-in, so the address is looked up once
// per device (with that device current) and cached.
sp_status scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return sp::report(SP_ERR_CUDA, "sp_select_noalloc: cudaGetDevice: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return sp::report(SP_ERR_UNSUPPORTED, "sp_select_noalloc: device ordinal %d", dev);
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_select_scratch);
    if (e != cudaSuccess || !p)
      return sp::report(SP_ERR_CUDA, "sp_select_noalloc: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
  return SP_OK;
}

}  // namespace

extern "C" sp_status sp_select_noalloc(const sp_selector* s, const sp_select_in* in, const sp_select_out* out,
                                       sp_stream stream) {
  const size_t need = sp_select_workspace(s, in);
  if (need == 0)  // invalid arguments: let the common path report the precise reason
    return sp::select_with_workspace(s, in, out, nullptr, 0, (cudaStream_t)stream);
  if (need > kScratchBytes)
    return sp::report(SP_ERR_WORKSPACE,
                      "sp_select_noalloc: this batch needs %zu bytes of scratch, more than the %zu-byte static "
                      "scratch; use sp_select with a caller workspace",
                      need, kScratchBytes);
  void* p = nullptr;
  sp_status st = scratch_address(&p);
  if (st != SP_OK) return st;
  // Nothing in the scratch is read before the same call writes it, so the
  // previous call's contents need no clearing.
  return sp::select_with_workspace(s, in, out, p, kScratchBytes, (cudaStream_t)stream);
}
