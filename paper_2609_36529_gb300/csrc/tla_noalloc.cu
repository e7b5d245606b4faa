// Forward entry point that allocates nothing: tla_chunk_fwd_noalloc.
//
// Some callers cannot call cudaMalloc at all, or not after start-up: plug-ins
// hosted by a runtime that owns every byte of device memory through its own
// pool, serving processes that forbid allocation on the request path to keep
// latency predictable, and code that must not grow the process's memory once a
// fixed budget has been committed.  Such a caller cannot provide the workspace
// tla_chunk_fwd needs, so this entry point uses a scratch buffer that is part
// of the library image itself: a file-scope device array of fixed size that
// every GPU which loads the library holds until the process exits.
//
// The caller still passes every input and output (p->o, p->ht).  Problems whose
// workspace exceeds the buffer are rejected on the host with
// TLA_ERR_WORKSPACE before anything is launched.  The buffer is shared by all
// calls and keeps whatever the last call left in it; the forward overwrites
// every scratch byte it reads, so nothing needs clearing, but two calls that
// overlap on the GPU (different streams, or different host threads without
// ordering) race on it.  The first call on each device looks up the buffer's
// device address (cudaGetSymbolAddress) with that device current; make that
// first call before capturing the stream into a CUDA graph.
#include <mutex>

#include "common.cuh"
#include "internal.h"

namespace tla {

// 64 MiB of scratch, 256-byte aligned (the workspace alignment the forward needs).
constexpr size_t kNoAllocScratchBytes = size_t(64) << 20;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of the scratch array on the current device (host code must not
// use the array's name as a device pointer).  Looked up once per device with that
// device current; a std::once_flag per device orders concurrent first calls.
constexpr int kMaxDevices = 64;
static tla_status noalloc_scratch(void** out) {
    static std::once_flag once[kMaxDevices];
    static void* addr[kMaxDevices] = {nullptr};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return TLA_ERR_CUDA;
    std::call_once(once[dev], [dev]() {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) == cudaSuccess) addr[dev] = p;
    });
    if (!addr[dev]) return TLA_ERR_CUDA;
    *out = addr[dev];
    return TLA_OK;
}

}  // namespace tla

using namespace tla;

extern "C" size_t tla_noalloc_scratch_bytes(void) { return kNoAllocScratchBytes; }

extern "C" tla_status tla_chunk_fwd_noalloc(const tla_problem* p, void* stream) {
    const size_t need = tla_fwd_workspace_bytes(p, 0);
    if (need == 0) {
        // invalid or unsupported problem: report the same status tla_chunk_fwd would
        return tla_chunk_fwd(p, nullptr, 0, 0, stream);
    }
    if (need > kNoAllocScratchBytes) return TLA_ERR_WORKSPACE;
    void* ws = nullptr;
    const tla_status st = noalloc_scratch(&ws);
    if (st != TLA_OK) return st;
    return tla_chunk_fwd(p, ws, kNoAllocScratchBytes, 0, stream);
}
