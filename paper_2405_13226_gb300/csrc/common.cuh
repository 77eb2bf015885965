// Shared device/host definitions of the attention kernels.
#pragma once
#include <cstdint>
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "ptx.cuh"

namespace ddattn {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// Device status codes (mirror dd_status in include/ddattn.h).
constexpr int kStatusTimeout = 5;

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

struct FwdParams {
  int B, L, H, nqt;
  float scale_log2;  // softmax scale * log2(e)
  const int32_t* offsets;
  int n_offsets;
  __nv_bfloat16* o;
  float* lse;
  int* status;
  unsigned long long timeout_ns;
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
  float* dq_acc;    // [B, H, L128, d] fp32
  __nv_bfloat16* dq;
  __nv_bfloat16* dk;
  __nv_bfloat16* dv;
  int* status;
  unsigned long long timeout_ns;
};

// Launchers (defined in attn_fwd.cu / attn_bwd.cu); return a cudaError_t.
cudaError_t launch_attn_fwd(int d, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                            const FwdParams& p, cudaStream_t stream);
cudaError_t launch_attn_bwd_main_d128(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                                      const CUtensorMap& tdo, const BwdParams& p, cudaStream_t stream);
cudaError_t launch_attn_bwd(int d, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                            const CUtensorMap& tdo, const BwdParams& p, int phases, cudaStream_t stream);

}  // namespace ddattn
