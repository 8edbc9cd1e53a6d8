// kvshot_static_ws.cu -- kvshot_draft_attn_static: draft attention whose
// scratch space is a fixed array of device memory built into this library,
// for callers that cannot allocate device memory themselves.
//
// The scratch is one file-scope __device__ array.  Every GPU that loads the
// library holds it (KVSHOT_STATIC_WORKSPACE_BYTES) until the process exits.
// In host code the array's name is only a host-side handle, never a device
// address, so the entry point looks the real address up once per device with
// cudaGetSymbolAddress (with that device current) and hands it to the
// ordinary attention path as its workspace.
#include <mutex>

#include "kvshot_internal.h"

namespace {

constexpr size_t kStaticBytes = KVSHOT_STATIC_WORKSPACE_BYTES;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_scratch[kStaticBytes];

void* g_scratch_addr[kMaxDevices] = {};
std::mutex g_scratch_mutex;

// Device address of g_scratch on the current device, looked up on the first
// call made with that device current.
kvshot_status scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return KVSHOT_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return KVSHOT_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || p == nullptr) return KVSHOT_ERR_CUDA;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return KVSHOT_OK;
}

}  // namespace

extern "C" kvshot_status kvshot_draft_attn_static(const kvshot_attn_desc* desc, const void* q, const void* target_k,
                                                  const void* target_v, const int32_t* page_table,
                                                  const int32_t* seq_lens, const void* draft_k, const void* draft_v,
                                                  const int32_t* tree_parent, void* out, float* lse,
                                                  kvshot_stream_t stream) {
  if (desc == nullptr) return KVSHOT_ERR_NULL;
  kvshot_attn_desc d = *desc;  // the caller's workspace fields are ignored
  d.workspace = nullptr;
  d.workspace_bytes = 0;
  const size_t need = kvshot_draft_attn_workspace_size(&d);
  if (need == 0) {
    // Invalid descriptor: let the ordinary entry point report the exact reason.
    return kvshot_draft_attn(&d, q, target_k, target_v, page_table, seq_lens, draft_k, draft_v, tree_parent, out,
                             lse, stream);
  }
  if (need > kStaticBytes) return KVSHOT_ERR_WORKSPACE;
  void* scratch = nullptr;
  if (kvshot_status st = scratch_address(&scratch)) return st;
  // The attention kernels write every scratch word they later read (each
  // piece's partial result before the merge reads it),
  // so nothing in the array has to be cleared between calls.
  d.workspace = scratch;
  d.workspace_bytes = kStaticBytes;
  return kvshot_draft_attn(&d, q, target_k, target_v, page_table, seq_lens, draft_k, draft_v, tree_parent, out, lse,
                           stream);
}
