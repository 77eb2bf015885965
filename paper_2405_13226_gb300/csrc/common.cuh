// Shared device/host definitions of the attention kernels.
#pragma once
#include <atomic>
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "../../include/ddattn.h"
#include "ptx.cuh"

namespace ddattn {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// Device status codes (mirror dd_status in include/ddattn.h).
constexpr int kStatusTimeout = 5;
constexpr int kStatusLayout = 6;

// Document start of token t (flattened index), per the document-mask rule:
// the largest offset <= t, never before the start of t's sequence
// (sequence boundaries always cut documents). offsets == nullptr: the
// sequence start. Clamped into [seq0, t] so malformed offsets cannot move
// any index out of the sequence.
__device__ __forceinline__ long long doc_start(const int32_t* off, int n, long long t, long long seq0) {
  if (off == nullptr) return seq0;
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if ((long long)__ldg(off + mid) <= t) lo = mid;
    else hi = mid - 1;
  }
  long long s = __ldg(off + lo);
  if (s > t) s = seq0;
  return s < seq0 ? seq0 : s;
}

// One past the last token of t's document: the first offset > t, never past
// the end of t's sequence. Clamped into [t + 1, seq_end].
__device__ __forceinline__ long long doc_end(const int32_t* off, int n, long long t, long long seq_end) {
  if (off == nullptr) return seq_end;
  int lo = 0, hi = n;  // first index with off[idx] > t, or n
  while (lo < hi) {
    int mid = (lo + hi) >> 1;
    if ((long long)__ldg(off + mid) > t) hi = mid;
    else lo = mid + 1;
  }
  long long e = lo < n ? (long long)__ldg(off + lo) : seq_end;
  if (e > seq_end) e = seq_end;
  return e <= t ? t + 1 : e;
}

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// Drain wait used only on the abort path: bounded by time, ignores the abort flag.
__device__ __forceinline__ void mbar_wait_drain(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > limit_ns) return;
  }
}

// RoPE frequencies theta_j = f_b^(-2j/d), j < d/2 <= 64, each split into an
// fp32 head and the fp32 rounding of its remainder (computed on the host in
// double precision).
struct RopeFreq {
  float hi[64], lo[64];
};

// (cos, sin) of m * theta_j for an integer position m < 2^24. The product is
// taken as p + e, p = fl(m * hi) and e = its exact rounding error (one fma)
// plus m * lo; sincosf gets the representable p, and the small e (|e| < ulp(p))
// is added by the angle-sum identity with cos e = 1 - e^2/2, sin e = e.
__device__ __forceinline__ float2 rope_cos_sin(int m, float hi, float lo) {
  const float fm = (float)m;
  const float p = fm * hi;
  float e = fmaf(fm, hi, -p);
  e = fmaf(fm, lo, e);
  float s, c;
  sincosf(p, &s, &c);
  const float h = 0.5f * e * e;
  return make_float2(fmaf(-e, s, fmaf(-h, c, c)), fmaf(e, c, fmaf(-h, s, s)));
}

// The backward's (cos, sin) table: one float4 (cos, sin of pair 2jj, cos, sin
// of pair 2jj + 1) per (position m, pair-pair jj), laid out
// [ceil(L/32)][d/4][32 positions] so that the 32 lanes of a warp, holding 32
// consecutive positions, read one contiguous 512-byte run for a given jj.
__device__ __forceinline__ long long rope_tab_index(int m, int d, int jj) {
  return ((long long)(m >> 5) * (d / 4) + jj) * 32 + (m & 31);
}

// R x for one pair (x0, x1) = (x_2j, x_2j+1) with (c, s) = (cos, sin) of m theta_j, fp32,
// rounded to a bf16 pair (first element in the low half). Every kernel that rotates q or k
// uses this, so they agree bit for bit.
__device__ __forceinline__ uint32_t rope_rotate_bf16x2(float x0, float x1, float c, float s) {
  return pack_bf16x2(fmaf(x0, c, -x1 * s), fmaf(x0, s, x1 * c));
}

// g <- R^T g for one rotated pair (cs = (cos, sin)).
__device__ __forceinline__ void rope_unrotate_pair(float& g0, float& g1, float c, float s) {
  const float a = fmaf(g0, c, g1 * s);
  const float b = fmaf(g1, c, -g0 * s);
  g0 = a;
  g1 = b;
}

// The first n (16 or 32) of 32 fp32 values -> bf16 at dst (16-byte aligned).
__device__ __forceinline__ void store_row(__nv_bfloat16* dst, const float (&f)[32], int n) {
  uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int q = 0; q < 4; q++) {
    if (8 * q >= n) break;
    d4[q] = make_uint4(pack_bf16x2(f[8 * q], f[8 * q + 1]), pack_bf16x2(f[8 * q + 2], f[8 * q + 3]),
                       pack_bf16x2(f[8 * q + 4], f[8 * q + 5]), pack_bf16x2(f[8 * q + 6], f[8 * q + 7]));
  }
}

// One slice of a dK row (n = 16 or 32 columns): dk = scale * acc, then R^T at
// position m when tab != nullptr (pair-pairs jj0 .. jj0 + n/4 - 1 of the table above).
__device__ __forceinline__ void store_dk_row32(__nv_bfloat16* dst, const uint32_t (&v)[32], float sc,
                                               const float4* tab, int m, int d, int jj0, int n) {
  float f[32];
#pragma unroll
  for (int e = 0; e < 32; e++) f[e] = __uint_as_float(v[e]) * sc;
  if (tab) {
#pragma unroll
    for (int u = 0; u < 8; u++) {
      if (4 * u >= n) break;
      const float4 cs = tab[rope_tab_index(m, d, jj0 + u)];
      rope_unrotate_pair(f[4 * u], f[4 * u + 1], cs.x, cs.y);
      rope_unrotate_pair(f[4 * u + 2], f[4 * u + 3], cs.z, cs.w);
    }
  }
  store_row(dst, f, n);
}

struct FwdParams {
  int B, L, H, nqt;
  float scale_log2;  // softmax scale * log2(e)
  const int32_t* offsets;
  int n_offsets;
  __nv_bfloat16* o;
  float* lse;
  int* status;
  unsigned int* work_ctr;  // items claimed past the first G (in the workspace's status block, zeroed per launch)
  unsigned long long timeout_ns;
  // RoPE forms only: rotated q / k written for the backward (with K tiles not rotated in
  // the kernel, k_rot is the k it reads, rotated by a pass before it), and the (cos, sin)
  // of m theta_j row-major [L, d/2] (in the workspace, filled before the kernel).
  __nv_bfloat16* q_rot;
  __nv_bfloat16* k_rot;
  const float2* rope_rows;
};

struct BwdParams {
  int B, L, H, L128, nkt;
  float scale, scale_log2;
  const int32_t* offsets;
  int n_offsets;
  const __nv_bfloat16* o;
  const __nv_bfloat16* dO;
  const float* lse;
  float* lse2_pad;  // [B, H, L128]: LSE * log2(e); +inf past L
  float* delta_pad; // [B, H, L128]: D_i = <dO_i, o_i>; 0 past L
  float* dq_acc;    // fp32: [B, H, L128, 64] for d = 64, else [B, H, ceil(d/32), L128, 32]
  __nv_bfloat16* dq;
  __nv_bfloat16* dk;
  __nv_bfloat16* dv;
  float4* rope_tab;       // (cos, sin) of m theta_j (layout of rope_tab_index), or nullptr without RoPE
  float2* rope_tab_rows;  // the same values row-major [L, d/2] (read where dq is written)
  RopeFreq rope;     // frequencies that fill rope_tab
  int dq_owned;      // the main kernel's CTAs own whole (sequence, head) pairs and write dq themselves
  int* status;
  unsigned long long timeout_ns;
};

struct RopeParams {
  long long rows;  // B * L token rows
  int L, H, d;
  const __nv_bfloat16* q;  // nullptr: rotate k only
  const __nv_bfloat16* k;
  __nv_bfloat16* q_rot;
  __nv_bfloat16* k_rot;
  RopeFreq f;
};

// One-time setup of a kernel per device: its dynamic shared-memory limit (a function
// attribute of each device's context, so set on every device the process launches on) and
// the device's SM count. `nsm` caches the count per device ordinal (0: not set up). The
// entries are atomics: host threads that race on a device's first launch both run the
// (idempotent) setup and store the same count.
constexpr int kMaxDevices = 64;
using DeviceCache = std::atomic<int>[kMaxDevices];
template <typename Kernel>
inline cudaError_t kernel_setup(DeviceCache& nsm, Kernel kernel, int smem_bytes, int* nsm_out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  int have = nsm[dev].load(std::memory_order_acquire);
  if (have == 0) {
    if (smem_bytes > 0 &&
        (e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes)) != cudaSuccess)
      return e;
    int n = 0;
    if ((e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    have = n < 1 ? 1 : n;
    nsm[dev].store(have, std::memory_order_release);
  }
  *nsm_out = have;
  return cudaSuccess;
}

// Host-side argument check of a descriptor (api.cu): DD_OK, DD_ERR_INVALID_ARG or
// DD_ERR_UNSUPPORTED, the code every entry point returns for that descriptor.
dd_status validate_desc(const dd_attn_desc* desc);

// Launchers (defined in attn_fwd.cu / attn_bwd.cu / rope.cu); return a cudaError_t.
// rope: 0 none; 1 the kernel rotates its Q tiles (k given rotated); 2 it rotates Q and K tiles.
cudaError_t launch_attn_fwd(int d, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                            const CUtensorMap& to, const FwdParams& p, int rope, cudaStream_t stream);
cudaError_t launch_attn_bwd_main_d128(int d, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                                      const CUtensorMap& tdo, const BwdParams& p, cudaStream_t stream);
cudaError_t launch_attn_bwd_main_d128_persist(int d, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                                      const CUtensorMap& tdo, const BwdParams& p, cudaStream_t stream);
cudaError_t launch_attn_bwd(int d, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                            const CUtensorMap& tdo, const BwdParams& p, int phases, cudaStream_t stream);
cudaError_t launch_rope_qk(const RopeParams& p, cudaStream_t stream);
cudaError_t launch_rope_table(int L, int d, const RopeFreq& f, float4* tab, float2* tab_rows, cudaStream_t stream);

}  // namespace ddattn
