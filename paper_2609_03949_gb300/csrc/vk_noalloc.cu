// vk_noalloc.cu -- vk_decode_step_noalloc: the decode step for callers that cannot provide a workspace.
//
// Some callers of this library cannot allocate device memory when they run a decode step: a plugin that a
// host program loads and that must use only memory the host handed to it, with no allocator reachable
// through a C interface; or a serving loop that fixed its device-memory budget at start-up and forbids any
// later cudaMalloc (which can also synchronise the device in the middle of the token loop). For them this
// entry point takes its scratch from one static device array instead of a caller-provided workspace.
//
// The array below is device memory that the CUDA runtime sets aside when it loads this library's code on a
// GPU (at the latest at this entry point's first call there) and keeps until the process exits. Its size is
// VK_NOALLOC_SCRATCH_BYTES; problems whose workspace (vk_workspace_bytes) is larger are rejected.
// Host code cannot use the array's name as a device address: the name is a host-side shadow. The device
// address is looked up with cudaGetSymbolAddress on every call, with the caller's device current: the lookup is
// cheap, and a cached address could outlive its module (after cudaDeviceReset the runtime loads the library's
// code again, and the array may then sit elsewhere).
#include <cstdio>

#include "vk_common.cuh"

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[VK_NOALLOC_SCRATCH_BYTES];

// Device address of g_noalloc_scratch on the current device, looked up afresh (the first lookup on a device
// loads the library's device code there if that has not happened yet).
cudaError_t scratch_address(void** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess) return e;
  *out = p;
  return cudaSuccess;
}

}  // namespace

namespace vk {
int record_error(int code, const char* msg);
}

extern "C" int vk_decode_step_noalloc(const vk_view* view, const vk_params* params, const vk_index* index,
                                      float* out, float* lse, float* smax, int32_t* idx, int32_t* count,
                                      int32_t cap, void* stream) {
  const size_t need = vk_workspace_bytes(view, params, cap);
  if (need == 0) {
    // invalid view or params: the workspace-taking entry point reports the precise refusal
    return vk_decode_step(view, params, index, out, lse, smax, idx, count, cap, nullptr, 0, stream);
  }
  if (need > (size_t)VK_NOALLOC_SCRATCH_BYTES) {
    char msg[160];
    snprintf(msg, sizeof(msg), "this problem needs %zu bytes of scratch; the static scratch holds %zu",
             need, (size_t)VK_NOALLOC_SCRATCH_BYTES);
    return vk::record_error(VK_ERR_WORKSPACE, msg);
  }
  void* scratch = nullptr;
  cudaError_t e = scratch_address(&scratch);
  if (e != cudaSuccess) return vk::record_error(VK_ERR_CUDA, cudaGetErrorString(e));
  // the array keeps the previous call's contents; the status word at its start must begin at zero
  e = cudaMemsetAsync(scratch, 0, 256, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return vk::record_error(VK_ERR_CUDA, cudaGetErrorString(e));
  return vk_decode_step(view, params, index, out, lse, smax, idx, count, cap, scratch,
                        (size_t)VK_NOALLOC_SCRATCH_BYTES, stream);
}
