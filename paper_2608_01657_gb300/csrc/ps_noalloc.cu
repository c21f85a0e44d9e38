// ps_cached_prefix_noalloc: the read-only cached-prefix probe for callers that
// cannot allocate device memory.
//
// ps_cached_prefix() keeps its per-call scratch (block offsets, hashing
// segments, per-position chain values, keys and lookup results) in the
// handle's workspace.  Some callers may not call cudaMalloc at all, or may not
// write into a workspace they do not own: code running inside a CUDA graph
// capture region, or inside a framework whose allocator owns every device
// allocation.  This entry point gives them the same answer with its scratch
// in one fixed, file-scope device array that the library holds for as long
// as it is loaded, on every GPU that loads it.  Only the scratch moves out of
// the workspace: the probe still reads the pool's table, which every ps_step()
// of the handle rewrites, so a probe must be stream-ordered against the
// handle's steps (an unordered probe could read a half-updated table).
#include <mutex>

#include "ps_internal.cuh"

namespace {

using namespace ps;

// Maximum sizes of one call: 4096 requests and 131072 full blocks.
constexpr int64_t kNaMaxRequests = 4096;
constexpr int64_t kNaMaxBlocks = 131072;
constexpr int64_t kNaMaxSegments = kNaMaxBlocks / kChunkBlocks + kNaMaxRequests + 1;

// Byte layout of the scratch array, every region 256-byte aligned.
constexpr size_t align256(size_t x) { return (x + 255) / 256 * 256; }
constexpr size_t kOffCtl = 0;
constexpr size_t kOffRq = align256(kOffCtl + sizeof(Ctl));
constexpr size_t kRqArrays = 5;  // n, h, s, fu, pbase
constexpr size_t kOffTile = align256(kOffRq + kRqArrays * align256(4 * kNaMaxRequests));
constexpr size_t kOffSeg = align256(kOffTile + 8 * (kNaMaxRequests / kValTile + 1));
constexpr size_t kOffPos = align256(kOffSeg + align256(sizeof(ChunkDesc) * kNaMaxSegments) + align256(8 * kNaMaxSegments));
constexpr size_t kScratchBytes = align256(kOffPos + align256(8 * kNaMaxBlocks) + 2 * align256(4 * kNaMaxBlocks));

// The scratch itself (about 2.4 MB).  In host code 'g_probe_scratch' names a
// host-side stand-in, not device memory: only the address returned by
// cudaGetSymbolAddress() may be handed to a kernel.
static __device__ __align__(256) unsigned char g_probe_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
unsigned char* g_scratch_ptr[kMaxDevices] = {};

// Once per device, with that device current: the device address of the array.
int32_t scratch_for_current_device(unsigned char** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return PS_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_probe_scratch) != cudaSuccess || !p) return PS_ERR_CUDA;
    g_scratch_ptr[dev] = static_cast<unsigned char*>(p);
  }
  *out = g_scratch_ptr[dev];
  return PS_OK;
}

}  // namespace

// The handle's layout is private to ps_api.cu; this file needs only its
// device state, which the first member of the handle holds.
struct ps_handle;
namespace ps {
const DevState* handle_state(const ps_handle_t* h);
}

extern "C" int32_t ps_cached_prefix_noalloc(ps_handle_t* h, void* stream, int32_t num_requests,
                                            const int32_t* d_group_ids, const int64_t* d_token_offsets,
                                            const int32_t* d_tokens, int32_t* d_cached_blocks, int32_t* d_status) {
  if (!h || num_requests < 0 || !d_token_offsets || !d_status) return PS_ERR_INVALID_ARG;
  // more requests than the handle takes: refused as by ps_cached_prefix();
  // more than the scratch array holds: a capacity error
  if (num_requests > handle_state(h)->max_requests) return PS_ERR_INVALID_ARG;
  if (num_requests > kNaMaxRequests) return PS_ERR_CAPACITY;
  if (num_requests > 0 && (!d_group_ids || !d_tokens || !d_cached_blocks)) return PS_ERR_INVALID_ARG;
  unsigned char* base = nullptr;
  const int32_t rc = scratch_for_current_device(&base);
  if (rc != PS_OK) return rc;
  DevState s = *handle_state(h);
  // bounds of one call: the smaller of the handle's and the scratch's
  s.max_requests = s.max_requests < kNaMaxRequests ? s.max_requests : (int32_t)kNaMaxRequests;
  if (s.max_blocks > kNaMaxBlocks) {
    s.max_blocks = kNaMaxBlocks;
    s.max_tokens = kNaMaxBlocks * s.bs;
  }
  s.max_segments = s.max_blocks / kChunkBlocks + s.max_requests + 1;
  // per-call scratch, carved from the static array
  const size_t rq = align256(4 * kNaMaxRequests);
  s.ctl = reinterpret_cast<Ctl*>(base + kOffCtl);
  s.rq_n = reinterpret_cast<int32_t*>(base + kOffRq + 0 * rq);
  s.rq_h = reinterpret_cast<int32_t*>(base + kOffRq + 1 * rq);
  s.rq_s = reinterpret_cast<int32_t*>(base + kOffRq + 2 * rq);
  s.rq_fu = reinterpret_cast<uint32_t*>(base + kOffRq + 3 * rq);
  s.rq_pbase = reinterpret_cast<int32_t*>(base + kOffRq + 4 * rq);
  s.val_tile = reinterpret_cast<uint64_t*>(base + kOffTile);
  s.chunks = reinterpret_cast<ChunkDesc*>(base + kOffSeg);
  s.seg_word = reinterpret_cast<uint64_t*>(base + kOffSeg + align256(sizeof(ChunkDesc) * kNaMaxSegments));
  s.pos_key = reinterpret_cast<uint64_t*>(base + kOffPos);
  s.pos_req = reinterpret_cast<uint32_t*>(base + kOffPos + align256(8 * kNaMaxBlocks));
  s.pos_blk = reinterpret_cast<uint32_t*>(base + kOffPos + align256(8 * kNaMaxBlocks) + align256(4 * kNaMaxBlocks));
  s.R = num_requests;
  s.in_group = d_group_ids;
  s.in_offsets = d_token_offsets;
  s.in_tokens = d_tokens;
  s.in_contract = nullptr;
  s.in_prefix = nullptr;
  s.tokens_aligned16 = (reinterpret_cast<uintptr_t>(d_tokens) & 15) == 0;
  // Every scratch word the probe reads it first writes in the same call (the
  // control block's per-call fields included), except validation's tile
  // totals and counters: those start at zero (a static array is zeroed at
  // load) and every call leaves them at zero, so nothing is cleared here.
  return launch_probe(s, reinterpret_cast<cudaStream_t>(stream), d_cached_blocks, d_status);
}
