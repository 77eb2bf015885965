// Host side of the C ABI declared in include/ddattn.h: argument checks,
// TMA tensor maps, workspace layout, launches and the device status word.
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstdlib>
#include <cudaTypedefs.h>

#include "../../include/ddattn.h"
#include "common.cuh"

namespace ddattn {
namespace {

constexpr size_t kStatusBytes = 256;  // status word + padding, keeps the rest 256-aligned

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

long long round128(long long L) { return (L + 127) / 128 * 128; }

dd_status check_desc(const dd_attn_desc* d) {
  if (!d) return DD_ERR_INVALID_ARG;
  if (d->B < 1 || d->L < 1 || d->H < 1) return DD_ERR_INVALID_ARG;
  if (d->B > 65535 || d->H > 65535) return DD_ERR_INVALID_ARG;  // grid y/z limits
  if (d->d != 64 && d->d != 80 && d->d != 128) return DD_ERR_UNSUPPORTED;
  if (!std::isfinite(d->scale) || !(d->scale > 0.f)) return DD_ERR_INVALID_ARG;
  if (d->cu_doc_offsets) {
    if (d->n_offsets < 2 || (reinterpret_cast<uintptr_t>(d->cu_doc_offsets) & 3u)) return DD_ERR_INVALID_ARG;
    if ((long long)d->B * d->L > 2147483647LL) return DD_ERR_INVALID_ARG;  // int32 offsets
  }
  if (!std::isfinite(d->rope_base) || d->rope_base < 0.f) return DD_ERR_INVALID_ARG;
  if (d->rope_base > 0.f && d->L > (1 << 24)) return DD_ERR_INVALID_ARG;  // positions exact in fp32
  return DD_OK;
}

bool has_rope(const dd_attn_desc* d) { return d->rope_base > 0.f; }

// theta_j = f_b^(-2j/d) in double, split into fp32 head + fp32 remainder.
RopeFreq rope_freq(const dd_attn_desc* d) {
  RopeFreq f{};
  for (int j = 0; j < d->d / 2; j++) {
    const double th = std::pow((double)d->rope_base, -2.0 * j / d->d);
    f.hi[j] = (float)th;
    f.lo[j] = (float)(th - (double)f.hi[j]);
  }
  return f;
}

size_t bwd_vec_bytes(const dd_attn_desc* d) {
  return align256((size_t)d->B * d->H * round128(d->L) * sizeof(float));
}
// fp32 dQ accumulator: [B, H, L128, 64] for d = 64, [B, H, ceil(d/32), L128, 32] otherwise.
size_t bwd_acc_bytes(const dd_attn_desc* d) {
  const size_t cols = d->d == 64 ? 64 : (size_t)(d->d + 31) / 32 * 32;
  return align256((size_t)d->B * d->H * round128(d->L) * cols * sizeof(float));
}
size_t rope_tab_bytes(const dd_attn_desc* d) {
  return has_rope(d) ? align256((size_t)((d->L + 31) / 32 * 32) * (d->d / 2) * sizeof(float2)) : 0;
}
size_t rope_rows_bytes(const dd_attn_desc* d) {
  return has_rope(d) ? align256((size_t)d->L * (d->d / 2) * sizeof(float2)) : 0;
}

// The driver's tensor-map encoder, looked up once (a function-local static initialised by
// its first caller; concurrent first callers wait for that initialisation).
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static const PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
  }();
  return fn;
}

// 4-D map over a [B, L, H, d] bf16 tensor (dims innermost first: d, H, L, B),
// box = 64 columns x 1 head x box_rows tokens x 1 sequence, 128B swizzle.
// Rows past L read as zeros.
bool make_map(CUtensorMap* m, const void* ptr, const dd_attn_desc* d, int box_rows) {
  auto enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[4] = {(cuuint64_t)d->d, (cuuint64_t)d->H, (cuuint64_t)d->L, (cuuint64_t)d->B};
  cuuint64_t strides[3] = {(cuuint64_t)d->d * 2, (cuuint64_t)d->H * d->d * 2,
                           (cuuint64_t)d->L * d->H * d->d * 2};
  cuuint32_t box[4] = {64, 1, (cuuint32_t)box_rows, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(ptr), dims, strides, box, es,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// The current device is an sm_103 part. The verdict is cached per device ordinal
// (0: not yet checked, 1: supported, 2: not), so host threads driving different GPUs
// each get their own device's answer.
dd_status check_device() {
  static std::atomic<int> verdict[kMaxDevices];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DD_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return DD_ERR_UNSUPPORTED;
  int v = verdict[dev].load(std::memory_order_acquire);
  if (v == 0) {
    int major = 0, minor = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
      return DD_ERR_CUDA;
    v = (major == 10 && minor == 3) ? 1 : 2;
    verdict[dev].store(v, std::memory_order_release);
  }
  return v == 1 ? DD_OK : DD_ERR_UNSUPPORTED;
}

// Bound of every device-side wait (DDATTN_WAIT_LIMIT_MS, default 1 s), read once.
unsigned long long wait_limit_ns() {
  static const unsigned long long v = [] {
    const char* e = std::getenv("DDATTN_WAIT_LIMIT_MS");
    long long ms = e ? std::atoll(e) : 1000;
    if (ms < 1) ms = 1;
    return (unsigned long long)ms * 1000000ull;
  }();
  return v;
}

// Sequences of at most this many key tiles (L <= 512) have their K tiles rotated inside the
// RoPE forward kernel: each K tile is loaded by at most two work items there. Longer ones
// load each K tile in many items, so k is rotated once by a pass before the kernel (measured
// per call at H = 16, d = 128, 65536 tokens: in-kernel K rotation 0.349 / 0.440 ms at
// L = 256 / 512 against 0.376 / 0.466 with the pass; 1.353 against 1.061 at 4096).
constexpr int kFwdRopeQKMaxTiles = 4;

dd_status fwd_common(const dd_attn_desc* desc, const void* q, const void* k, const void* v, void* o, float* lse,
                     void* q_rot, void* k_rot, void* ws, size_t ws_bytes, void* stream, bool fused_rope) {
  dd_status st = check_desc(desc);
  if (st != DD_OK) return st;
  if (!q || !k || !v || !o || !lse) return DD_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(lse))
    return DD_ERR_INVALID_ARG;
  if (fused_rope) {
    if (!has_rope(desc) || !q_rot || !k_rot || !aligned16(q_rot) || !aligned16(k_rot)) return DD_ERR_INVALID_ARG;
    const uintptr_t kb = reinterpret_cast<uintptr_t>(k), kr = reinterpret_cast<uintptr_t>(k_rot);
    const uintptr_t n = (uintptr_t)desc->B * desc->L * desc->H * desc->d * 2;
    if (kr < kb + n && kb < kr + n) return DD_ERR_INVALID_ARG;  // k_rot must not overlap k
  }
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < dd_attn_workspace_size(desc, 0))
    return DD_ERR_WORKSPACE;
  if ((st = check_device()) != DD_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int nkt = (desc->L + 127) / 128;
  const int rope = !fused_rope ? 0 : (nkt <= kFwdRopeQKMaxTiles ? 2 : 1);  // launch_attn_fwd's RoPE form
  CUtensorMap tq, tk, tv, to;
  if (!make_map(&tq, q, desc, 128) || !make_map(&tk, rope == 1 ? k_rot : k, desc, 128) ||
      !make_map(&tv, v, desc, 128) || !make_map(&to, o, desc, 32))  // o: stored in 32-row blocks
    return DD_ERR_CUDA;
  FwdParams p;
  p.B = desc->B;
  p.L = desc->L;
  p.H = desc->H;
  p.nqt = nkt;
  p.scale_log2 = desc->scale * kLog2e;
  p.offsets = desc->cu_doc_offsets;
  p.n_offsets = desc->cu_doc_offsets ? desc->n_offsets : 0;
  p.o = static_cast<__nv_bfloat16*>(o);
  p.lse = lse;
  p.status = static_cast<int*>(ws);
  p.work_ctr = reinterpret_cast<unsigned int*>(static_cast<uint8_t*>(ws) + 64);  // inside the status block
  p.timeout_ns = wait_limit_ns();
  p.q_rot = static_cast<__nv_bfloat16*>(q_rot);
  p.k_rot = static_cast<__nv_bfloat16*>(k_rot);
  p.rope_rows = nullptr;
  cudaError_t e = cudaSuccess;
  if (fused_rope) {
    float2* rows = reinterpret_cast<float2*>(static_cast<uint8_t*>(ws) + kStatusBytes);
    p.rope_rows = rows;
    const RopeFreq f = rope_freq(desc);
    if ((e = launch_rope_table(desc->L, desc->d, f, nullptr, rows, s)) != cudaSuccess) return DD_ERR_CUDA;
    if (rope == 1) {  // k -> k_rot in one pass; the kernel reads k_rot
      RopeParams rp;
      rp.rows = (long long)desc->B * desc->L;
      rp.L = desc->L;
      rp.H = desc->H;
      rp.d = desc->d;
      rp.q = nullptr;
      rp.k = static_cast<const __nv_bfloat16*>(k);
      rp.q_rot = nullptr;
      rp.k_rot = static_cast<__nv_bfloat16*>(k_rot);
      rp.f = f;
      if ((e = launch_rope_qk(rp, s)) != cudaSuccess) return DD_ERR_CUDA;
    }
  }
  e = launch_attn_fwd(desc->d, tq, tk, tv, to, p, rope, s);
  return e == cudaSuccess ? DD_OK : DD_ERR_CUDA;
}

}  // namespace

dd_status validate_desc(const dd_attn_desc* desc) { return check_desc(desc); }

// One warp waits on an mbarrier that nothing arrives on; the bounded wait
// expires after limit_ns and records the timeout in *status.
__global__ void selftest_wait_kernel(int* status, unsigned long long limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    abort_flag = 0;
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  Watchdog wd{&abort_flag, status, limit_ns};
  (void)mbar_wait(&bar, 0, wd);
}

}  // namespace ddattn

using namespace ddattn;

extern "C" {

size_t dd_attn_workspace_size(const dd_attn_desc* desc, int for_bwd) {
  if (check_desc(desc) != DD_OK) return 0;
  if (!for_bwd) return kStatusBytes + rope_rows_bytes(desc);  // + the RoPE forward's (cos, sin) rows
  return kStatusBytes + 2 * bwd_vec_bytes(desc) + bwd_acc_bytes(desc) + rope_tab_bytes(desc) + rope_rows_bytes(desc);
}

dd_status dd_rope_qk(const dd_attn_desc* desc, const void* q, const void* k, void* q_rot, void* k_rot,
                     void* stream) {
  dd_status st = check_desc(desc);
  if (st != DD_OK) return st;
  if (!has_rope(desc)) return DD_ERR_INVALID_ARG;
  if (!q || !k || !q_rot || !k_rot) return DD_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(q_rot) || !aligned16(k_rot)) return DD_ERR_INVALID_ARG;
  if ((st = check_device()) != DD_OK) return st;
  RopeParams p;
  p.rows = (long long)desc->B * desc->L;
  p.L = desc->L;
  p.H = desc->H;
  p.d = desc->d;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.k = static_cast<const __nv_bfloat16*>(k);
  p.q_rot = static_cast<__nv_bfloat16*>(q_rot);
  p.k_rot = static_cast<__nv_bfloat16*>(k_rot);
  p.f = rope_freq(desc);
  return launch_rope_qk(p, static_cast<cudaStream_t>(stream)) == cudaSuccess ? DD_OK : DD_ERR_CUDA;
}

dd_status dd_attn_fwd(const dd_attn_desc* desc, const void* q, const void* k, const void* v, void* o, float* lse,
                      void* ws, size_t ws_bytes, void* stream) {
  return fwd_common(desc, q, k, v, o, lse, nullptr, nullptr, ws, ws_bytes, stream, false);
}

dd_status dd_attn_fwd_rope(const dd_attn_desc* desc, const void* q, const void* k, const void* v, void* o,
                           float* lse, void* q_rot, void* k_rot, void* ws, size_t ws_bytes, void* stream) {
  return fwd_common(desc, q, k, v, o, lse, q_rot, k_rot, ws, ws_bytes, stream, true);
}

dd_status dd_attn_bwd(const dd_attn_desc* desc, const void* q, const void* k, const void* v, const void* o,
                      const void* dO, const float* lse, void* dq, void* dk, void* dv, void* ws, size_t ws_bytes,
                      void* stream) {
  return dd_attn_bwd_phases(desc, q, k, v, o, dO, lse, dq, dk, dv, ws, ws_bytes, DD_BWD_ALL, stream);
}

dd_status dd_attn_bwd_phases(const dd_attn_desc* desc, const void* q, const void* k, const void* v,
                             const void* o, const void* dO, const float* lse, void* dq, void* dk, void* dv,
                             void* ws, size_t ws_bytes, int phases, void* stream) {
  if (phases < 1 || phases > DD_BWD_ALL) return DD_ERR_INVALID_ARG;
  dd_status st = check_desc(desc);
  if (st != DD_OK) return st;
  if (!q || !k || !v || !o || !dO || !lse || !dq || !dk || !dv) return DD_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(dO) || !aligned16(lse) ||
      !aligned16(dq) || !aligned16(dk) || !aligned16(dv))
    return DD_ERR_INVALID_ARG;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u) || ws_bytes < dd_attn_workspace_size(desc, 1))
    return DD_ERR_WORKSPACE;
  if ((st = check_device()) != DD_OK) return st;
  const int bq = 128;  // query rows per backward step (both head dims)
  CUtensorMap tq, tk, tv, tdo;
  if (!make_map(&tq, q, desc, bq) || !make_map(&tk, k, desc, 128) || !make_map(&tv, v, desc, 128) ||
      !make_map(&tdo, dO, desc, bq))
    return DD_ERR_CUDA;
  uint8_t* w = static_cast<uint8_t*>(ws);
  BwdParams p;
  p.B = desc->B;
  p.L = desc->L;
  p.H = desc->H;
  p.L128 = (int)round128(desc->L);
  p.nkt = (desc->L + 127) / 128;
  p.scale = desc->scale;
  p.scale_log2 = desc->scale * kLog2e;
  p.offsets = desc->cu_doc_offsets;
  p.n_offsets = desc->cu_doc_offsets ? desc->n_offsets : 0;
  p.o = static_cast<const __nv_bfloat16*>(o);
  p.dO = static_cast<const __nv_bfloat16*>(dO);
  p.lse = lse;
  p.lse2_pad = reinterpret_cast<float*>(w + kStatusBytes);
  p.delta_pad = reinterpret_cast<float*>(w + kStatusBytes + bwd_vec_bytes(desc));
  p.dq_acc = reinterpret_cast<float*>(w + kStatusBytes + 2 * bwd_vec_bytes(desc));
  p.dq = static_cast<__nv_bfloat16*>(dq);
  p.dk = static_cast<__nv_bfloat16*>(dk);
  p.dv = static_cast<__nv_bfloat16*>(dv);
  uint8_t* rope_base = w + kStatusBytes + 2 * bwd_vec_bytes(desc) + bwd_acc_bytes(desc);
  p.rope_tab = has_rope(desc) ? reinterpret_cast<float4*>(rope_base) : nullptr;
  p.rope_tab_rows = has_rope(desc) ? reinterpret_cast<float2*>(rope_base + rope_tab_bytes(desc)) : nullptr;
  p.rope = has_rope(desc) ? rope_freq(desc) : RopeFreq{};
  p.dq_owned = 0;  // chosen by the launcher from the key-tile count
  p.status = static_cast<int*>(ws);
  p.timeout_ns = wait_limit_ns();
  cudaError_t e = launch_attn_bwd(desc->d, tq, tk, tv, tdo, p, phases, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? DD_OK : DD_ERR_CUDA;
}

dd_status dd_selftest_wait_timeout(void* ws, uint32_t limit_us, void* stream) {
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255u)) return DD_ERR_WORKSPACE;
  if (limit_us < 1 || limit_us > 1000000) return DD_ERR_INVALID_ARG;
  selftest_wait_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(static_cast<int*>(ws),
                                                                        (unsigned long long)limit_us * 1000ull);
  return cudaGetLastError() == cudaSuccess ? DD_OK : DD_ERR_CUDA;
}

dd_status dd_attn_clear_status(void* ws, void* stream) {
  if (!ws) return DD_ERR_WORKSPACE;
  return cudaMemsetAsync(ws, 0, sizeof(int), static_cast<cudaStream_t>(stream)) == cudaSuccess ? DD_OK
                                                                                             : DD_ERR_CUDA;
}

dd_status dd_attn_poll_status(const void* ws) {
  if (!ws) return DD_ERR_WORKSPACE;
  if (cudaDeviceSynchronize() != cudaSuccess) return DD_ERR_CUDA;
  int v = 0;
  if (cudaMemcpy(&v, ws, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return DD_ERR_CUDA;
  return static_cast<dd_status>(v);
}

const char* dd_status_string(dd_status s) {
  switch (s) {
    case DD_OK: return "ok";
    case DD_ERR_INVALID_ARG: return "invalid argument";
    case DD_ERR_UNSUPPORTED: return "unsupported (head dim must be 64, 80 or 128; device must be sm_103)";
    case DD_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case DD_ERR_CUDA: return "CUDA runtime error";
    case DD_ERR_DEVICE_TIMEOUT: return "device-side wait timed out";
    case DD_ERR_DEVICE_LAYOUT: return "kernel shared-memory base misaligned (nothing computed)";
  }
  return "unknown status";
}

}  // extern "C"
