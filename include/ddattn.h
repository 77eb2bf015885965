/*
 * ddattn.h -- C ABI of libddattn.so: causal / document-masked multi-head
 * self-attention, forward and backward, for one training step on one GPU
 * (hand-written sm_103a kernels: TMA, tcgen05 UMMA, TMEM accumulators).
 *
 * The operation (Sec. 2.2 "Variable sequence length training" and Sec. 1):
 *   a step is B sequences of one length L. Under dataset decomposition every
 *   sequence is cut from a single document (Sec. 2.1, property (2)), so the
 *   mask is plain causal (query i attends to keys j <= i). Under the
 *   concat-and-chunk baseline with document masking (Sec. 1, Sec. 3.5 "DM"),
 *   a chunk holds several documents and query i only attends to keys j <= i
 *   of its own document; cu_doc_offsets gives the document starts.
 *   With s_ij = scale * <q_i, k_j> over the live keys A(i):
 *     LSE_i = ln sum_{j in A(i)} exp(s_ij),  P_ij = exp(s_ij - LSE_i),
 *     o_i = sum_j P_ij v_j.
 *   Backward, given dO = dLoss/do:
 *     D_i = <dO_i, o_i>, dS_ij = P_ij (<dO_i, v_j> - D_i),
 *     dq_i = scale sum_j dS_ij k_j, dk_j = scale sum_i dS_ij q_i,
 *     dv_j = sum_i P_ij dO_i.
 *
 * Rotary position embedding (Sec. 3, training setup; base frequency f_b of
 * the f_b ablation table and Table 2): before attention, consecutive
 * components of every q and k head vector are rotated by the token's position
 * m inside its sequence,
 *     theta_j = f_b^(-2j/d),
 *     (x_2j, x_2j+1) -> (x_2j cos m theta_j - x_2j+1 sin m theta_j,
 *                        x_2j sin m theta_j + x_2j+1 cos m theta_j).
 *   dd_attn_fwd_rope applies it inside the forward kernel and also returns the
 *   rotated q and k; dd_rope_qk applies it as a separate pass (bf16 out). With
 *   desc->rope_base = f_b > 0, the q and k given to dd_attn_fwd / dd_attn_bwd
 *   are the ROTATED ones, and
 *   dd_attn_bwd returns dq, dk with respect to the UN-rotated q and k (it
 *   applies the transposed rotation to the rotated-space gradients inside its
 *   kernels). rope_base = 0 means no rotation.
 *
 * Layouts (all device memory, caller-owned, never freed or kept by the library):
 *   q, k, v, o, dO, dq, dk, dv : bf16, [B, L, H, d] contiguous (token-major).
 *   lse                        : fp32, [B, H, L] contiguous, natural log.
 *   cu_doc_offsets             : int32 [n_offsets], document starts over the
 *                                flattened B*L tokens, non-decreasing, first 0,
 *                                last B*L. Sequence boundaries b*L always cut
 *                                documents, listed or not. NULL = plain causal.
 *   ws                         : workspace of dd_attn_workspace_size() bytes,
 *                                256-byte aligned. Its first 256 bytes are a
 *                                status block: the device status word in the
 *                                first 16 bytes (zero it once before first use,
 *                                dd_attn_clear_status) and the forward's
 *                                work-item counter at byte 64 (each forward call
 *                                zeroes it on its stream). fwd and bwd may share
 *                                one workspace sized for bwd; calls that share a
 *                                workspace must not overlap on the GPU.
 * All data pointers must be 16-byte aligned. Calls are asynchronous and
 * ordered on `stream` (a cudaStream_t; NULL = legacy default stream).
 *
 * Errors: argument checks run on the host before any launch and return
 * DD_ERR_INVALID_ARG / DD_ERR_UNSUPPORTED / DD_ERR_WORKSPACE with nothing
 * launched. A failed launch returns DD_ERR_CUDA. Every wait inside the
 * kernels is bounded; a wait that expires ends the kernel and records
 * DD_ERR_DEVICE_TIMEOUT in the workspace status word (dd_attn_poll_status).
 * A backward kernel whose dynamic shared memory does not start 1024-aligned
 * (never seen on sm_103) records DD_ERR_DEVICE_LAYOUT there and returns.
 * Offsets that break the rules above give undefined values but no
 * out-of-bounds access: every derived index is clamped into the sequence.
 */
#ifndef DDATTN_H
#define DDATTN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  DD_OK = 0,
  DD_ERR_INVALID_ARG = 1,     /* null / misaligned pointer, bad sizes */
  DD_ERR_UNSUPPORTED = 2,     /* head dim other than 64, 80 or 128, device not sm_103 */
  DD_ERR_WORKSPACE = 3,       /* workspace missing or smaller than required */
  DD_ERR_CUDA = 4,            /* a CUDA runtime call or launch failed */
  DD_ERR_DEVICE_TIMEOUT = 5,  /* a bounded device-side wait expired */
  DD_ERR_DEVICE_LAYOUT = 6    /* a kernel found its shared-memory base misaligned and did nothing */
} dd_status;

typedef struct {
  int32_t B;                       /* sequences per call (>= 1) */
  int32_t L;                       /* tokens per sequence (>= 1; multiples of 128 are the fast path) */
  int32_t H;                       /* heads (>= 1) */
  int32_t d;                       /* head dim: 64, 80 (OpenLM-3B heads) or 128 */
  float scale;                     /* softmax scale, usually 1/sqrt(d); finite */
  const int32_t* cu_doc_offsets;   /* DEVICE pointer or NULL (plain causal) */
  int32_t n_offsets;               /* entries of cu_doc_offsets (>= 2 when non-NULL) */
  float rope_base;                 /* RoPE base frequency f_b; 0 = no RoPE; else finite and > 0 */
} dd_attn_desc;

/* Workspace bytes for dd_attn_fwd / dd_attn_fwd_rope (for_bwd = 0) or
 * dd_attn_bwd (for_bwd = 1): the status word, for fwd with rope_base > 0 the
 * fp32 (cos, sin) table [L, d/2] of dd_attn_fwd_rope, and for bwd the fp32 dQ accumulator (B*H*L128*d' floats,
 * d' = 64 for d = 64, else d rounded up to a multiple of 32) plus
 * the per-row D_i and LSE_i*log2(e) vectors [B, H, L128], L128 = L rounded up
 * to a multiple of 128, plus, when rope_base > 0, two copies of the
 * (cos, sin) table of every position and pair (fp32, (L rounded up to 32 +
 * L) * d/2 pairs). Returns 0 for an invalid descriptor. */
size_t dd_attn_workspace_size(const dd_attn_desc* desc, int for_bwd);

/* Forward (Sec. 2.2 step; mask per cu_doc_offsets): writes o and lse. One CTA
 * per SM walks the work items (two 128-row query tiles of one sequence and
 * head), claiming each next one from the counter in the workspace's status
 * block; a memset of that counter precedes the kernel on `stream`. */
dd_status dd_attn_fwd(const dd_attn_desc* desc, const void* q, const void* k, const void* v, void* o, float* lse,
                      void* ws, size_t ws_bytes, void* stream);

/* Rotary position embedding of q and k (see the top of this file): writes
 * q_rot = R q and k_rot = R k, bf16, [B, L, H, d] like q and k, computed in
 * fp32 from the bf16 inputs and rounded to nearest-even. Needs
 * desc->rope_base > 0; the mask fields of desc are ignored (positions restart
 * at every sequence, not at every document: RoPE scores depend on m - n only,
 * so inside a document the two choices agree). In place (q_rot == q,
 * k_rot == k) is allowed. One bandwidth-bound kernel, no workspace. */
dd_status dd_rope_qk(const dd_attn_desc* desc, const void* q, const void* k, void* q_rot, void* k_rot,
                     void* stream);

/* Forward with the RoPE rotation fused into the kernel (the rotation above;
 * Sec. 3 training setup, RoPE base f_b of the f_b ablation table and Table 2):
 * q and k are the UN-rotated projections. Each 128-row Q tile is loaded once
 * per forward; the kernel rotates it in shared memory right after its TMA copy
 * lands and before the tensor core reads it, and writes it to q_rot. For
 * sequences of at most 4 key tiles (L <= 512) it does the same with every K
 * tile it loads, and each K tile reaches k_rot from the work item on whose
 * diagonal it lies. Longer sequences load each K tile in many work items, so
 * their k is rotated once, into k_rot, by a bandwidth-bound pass on `stream`
 * before the kernel, which then reads k_rot. The arithmetic is dd_rope_qk's
 * (fp32, bf16 rounding); the kernel steps the (cos, sin) of a row from the
 * position table by an angle-sum step of 8 positions, so a rotated value can
 * differ from dd_rope_qk's in its last bit (rarely). Outputs: o, lse and
 * q_rot = R q, k_rot = R k (bf16, [B, L, H, d]), the q and k that dd_attn_bwd
 * takes with rope_base > 0. Needs desc->rope_base > 0 and
 * dd_attn_workspace_size(desc, 0) bytes of workspace (this call fills the
 * table in it). q_rot may be q (in place); k_rot must not overlap k
 * (DD_ERR_INVALID_ARG): work items still read k while others write k_rot. */
dd_status dd_attn_fwd_rope(const dd_attn_desc* desc, const void* q, const void* k, const void* v, void* o,
                           float* lse, void* q_rot, void* k_rot, void* ws, size_t ws_bytes, void* stream);

/* Backward: from q, k, v, the forward's o and lse, and dO, writes dq, dk, dv
 * (bf16, overwritten, not accumulated). Recomputes P from lse. With
 * rope_base > 0, q and k are the rotated ones and dq, dk are returned with
 * respect to the un-rotated q, k. */
dd_status dd_attn_bwd(const dd_attn_desc* desc, const void* q, const void* k, const void* v, const void* o,
                      const void* dO, const float* lse, void* dq, void* dk, void* dv, void* ws, size_t ws_bytes,
                      void* stream);

/* The backward as its three kernels, for callers that time or schedule them
 * separately: DD_BWD_PRE (D_i, padded LSE, zero the dQ accumulator in ws),
 * DD_BWD_MAIN (P recompute and the five contractions; dK, dV and the fp32 dQ
 * accumulator), DD_BWD_POST (dq = bf16(scale * accumulator)). With RoPE the
 * PRE phase also fills the (cos, sin) table, and MAIN / POST rotate dk / dq
 * back with it. For sequences of at most 256 tokens at d = 80 / 128, MAIN
 * writes dq itself (its CTAs own whole (sequence, head) pairs and keep their
 * fp32 dQ rows in the accumulator, one region per CTA), PRE does not zero the
 * accumulator and POST launches nothing. `phases` is a
 * bit mask; issuing the phases in this order, with the same arguments and
 * workspace, equals one dd_attn_bwd call (dd_attn_bwd = all three). */
enum { DD_BWD_PRE = 1, DD_BWD_MAIN = 2, DD_BWD_POST = 4, DD_BWD_ALL = 7 };
dd_status dd_attn_bwd_phases(const dd_attn_desc* desc, const void* q, const void* k, const void* v,
                             const void* o, const void* dO, const float* lse, void* dq, void* dk, void* dv,
                             void* ws, size_t ws_bytes, int phases, void* stream);

/* Backward for callers that cannot allocate device memory: a runtime whose
 * own allocator holds all device memory and passes this library only the
 * tensors it owns, or a step loop under a fixed memory budget where a
 * cudaMalloc at step time is not allowed. The paper has no counterpart; this
 * is a library convenience. Same operation and arguments as dd_attn_bwd, but
 * no workspace: it uses a scratch array of DD_NOALLOC_SCRATCH_BYTES that the
 * library keeps in device global memory (every GPU that loads the library
 * holds it until the process exits). Sizes whose bwd workspace
 * (dd_attn_workspace_size(desc, 1)) exceeds that return DD_ERR_WORKSPACE with
 * nothing launched; a bad descriptor returns the same code as dd_attn_bwd.
 * It calls no cudaMalloc / cudaFree. The first call on a device looks up the
 * array's device address (make it before any stream capture); that address
 * belongs to the device's context, so do not use this entry point on a device
 * after cudaDeviceReset in the same process. All calls share the array: calls
 * whose kernels overlap on the GPU race, so order them on one stream.
 * device_status (device memory, may be NULL) receives this call's device
 * status word (0, DD_ERR_DEVICE_TIMEOUT or DD_ERR_DEVICE_LAYOUT), copied on
 * `stream` after the backward. */
#define DD_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)
dd_status dd_attn_bwd_noalloc(const dd_attn_desc* desc, const void* q, const void* k, const void* v,
                              const void* o, const void* dO, const float* lse, void* dq, void* dk, void* dv,
                              int32_t* device_status, void* stream);

/* Zero the device status word at the head of `ws` (stream-ordered). */
dd_status dd_attn_clear_status(void* ws, void* stream);

/* Synchronise the device and return the device status word of `ws`
 * (DD_OK, or the first error a kernel recorded there). */
dd_status dd_attn_poll_status(const void* ws);

/* Self-test of the device-side failure path: launches one warp that waits,
 * with the same bounded wait the attention kernels use, on an mbarrier that
 * nothing ever arrives on. After `limit_us` microseconds the wait gives up,
 * the warp records DD_ERR_DEVICE_TIMEOUT in the status word of `ws` and the
 * kernel returns normally (no trap, the context stays usable). Returns
 * DD_ERR_CUDA if the launch fails, else DD_OK; read the outcome with
 * dd_attn_poll_status. limit_us must be in [1, 1000000]. */
dd_status dd_selftest_wait_timeout(void* ws, uint32_t limit_us, void* stream);

/* Static description of a status code. */
const char* dd_status_string(dd_status s);

#ifdef __cplusplus
}
#endif
#endif /* DDATTN_H */
