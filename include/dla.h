/*
 * dla.h -- C ABI of the GB300 (sm_103a) Dynamic Linear Attention forward path
 * (DLA, arXiv 2606.10650).
 *
 * The library computes, per (batch b, head h) stream, the multi-state linear
 * attention of the paper:
 *   - Information-Aware Dynamic State Merging (Sec. 3.1, Algorithm 1): each
 *     token state s_t = v_t k_t^T is scored against the most recent state S,
 *     I_t = ||N(s_t) - N(S)||_F / (||N(S)||_F + eps) with N the whole-matrix
 *     RMSNorm (gain 1); b_t = 1[I_t >= tau] opens a new state, otherwise the
 *     token is added to the open state (Sec. 3.1 update rule);
 *   - Capacity-Bounded Memory Modeling (Sec. 3.2, Algorithm 2): a
 *     chronologically ordered cache of at most C states; before appending to a
 *     full cache the adjacent pair i* = argmin (Ibar_i + Ibar_{i+1}) /
 *     (n_i + n_{i+1}) is merged (S, n and Ibar summed, the rest shifted);
 *   - the read-out (Eq. capacity_bounded_output):
 *     o_t = sum_{i < m_t} lambda_{t,i} S_i q_t over the cache after token t.
 *
 * Conventions
 *   - Every pointer argument is DEVICE memory owned by the caller, except the
 *     dla_params / dla_cache structs themselves, which are read on the host,
 *     and the q, k, v, lam, o of dla_forward_host, which are host memory.
 *     The library never allocates device memory and frees nothing.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  All device
 *     work is enqueued asynchronously on it; argument errors are returned
 *     synchronously before anything is enqueued.  A launch failure returns
 *     DLA_ERR_CUDA.  No C++ exception crosses this interface.
 *   - Failures found on the device -- a bounded wait of a kernel that gave up
 *     (DLA_ERR_TIMEOUT) or an inconsistent cache or snapshot list
 *     (DLA_ERR_DEVICE_CHECK) -- cannot be returned by the call that enqueued
 *     the work.  Each call folds its device status into a status word of its
 *     stream (the first failure since the last read sticks), and
 *     dla_sync_status(stream) waits for the stream and returns that status.
 *     dla_forward also leaves its own call's status in its workspace.  After a
 *     device failure the call's outputs and cache are undefined; the library
 *     stays usable (every wait is bounded, no kernel traps).  Two environment
 *     variables, read at every call and unset in normal use, exist for tests
 *     of this path: DLA_DEBUG_WAIT_MS=x makes every bounded wait give up after
 *     about x ms instead of about 2 s, and DLA_DEBUG_WITHHOLD_PIECES=1 makes
 *     dla_forward_host report only its first input piece as arrived.
 *   - The first call on each device from each host thread creates that
 *     thread's internal streams and events and looks up the device address
 *     of the library's status words; make it before any stream capture.
 *   - Layouts are row-major and contiguous:
 *       q, k, v   [B, T, H, d]   (bf16 or fp32, see dla_dtype)
 *       lambda    [B, T, H, C]   fp32, logical cache slot i = 0 is the oldest
 *                                state; entries i >= m_t are ignored;
 *                                NULL means every lambda is 1 (Algorithm 2's
 *                                un-weighted sum)
 *       o         [B, T, H, d]   fp32 or bf16 (dla_params.out_dtype)
 *       boundary  [B, H, T]      uint8, b_t (the first token of an empty
 *                                cache is reported as 1)
 *       merge_log [B, H, T]      int32, i* of the merge at token t, else -1
 *   - States are d_v x d_k matrices S = sum_s v_s k_s^T (the recurrent form of
 *     Sec. 2), stored row-major [d_v][d_k].
 *   - Supported: d_k = d_v = d in {64, 128}; 2 <= C <= 64; T >= 1.  Anything
 *     else returns DLA_ERR_UNSUPPORTED (shape outside the built kernels) or
 *     DLA_ERR_INVALID_ARG (meaningless value).
 *   - DLA(I), dynamic state merging without the capacity bound (Table 5): a
 *     capacity C that no stream's segment count reaches gives exactly its
 *     results.  dla_forward and dla_forward_noalloc also take 64 < C <= 256
 *     for bf16 inputs with d = 128 over whole rows of device-resident inputs
 *     (no seq_lens, no packed rows, not dla_forward_host); those instances hold
 *     no capacity merge, so a stream whose segment count would pass C fails
 *     the call's device check (DLA_ERR_DEVICE_CHECK, results undefined).
 *     dla_decode_step and dla_backward take C <= 64.
 */
#ifndef DLA_H
#define DLA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DLA_VERSION 4

typedef enum {
  DLA_OK = 0,
  DLA_ERR_INVALID_ARG = 1,  /* NULL where a pointer is required, bad value   */
  DLA_ERR_UNSUPPORTED = 2,  /* shape/dtype outside the built kernels         */
  DLA_ERR_WORKSPACE = 3,    /* workspace NULL or smaller than required       */
  DLA_ERR_CUDA = 4,         /* a CUDA runtime call or launch failed          */
  DLA_ERR_TIMEOUT = 5,      /* a bounded device wait gave up                 */
  DLA_ERR_DEVICE_CHECK = 6  /* a device-side consistency check failed        */
} dla_status;

typedef enum { DLA_BF16 = 0, DLA_F32 = 1 } dla_dtype;

/* Method parameters (Sec. 3.1 / 3.2).  Defaults (dla_default_params): tau 0.6
 * and capacity 30 are the paper's defaults (Sec. 4 ablation / Sec. 4.1);
 * eps = rms_eps = 1e-6.
 *   score_mode 0: Algorithm 1's score, token state s_t against the last state.
 *   score_mode 1: Eq. (importance_score) read literally: N(S + s_t) against N(S).
 *   from_cache  0: dla_forward starts from an empty cache (prefill);
 *               1: it continues from the contents of `cache` (chunked prefill).
 *   seq_lens    NULL: every batch row holds T tokens.  Else device int32 [B],
 *               4-byte aligned (ragged batches in the padded layout): row b
 *               holds its first seq_lens[b] tokens (clamped to [0, T]); the
 *               tokens after them are padding: not processed, boundary 0 and
 *               merge_log -1 there, their o rows not written, and the row's
 *               cache is the one after its own tokens.  The forward calls read
 *               it; dla_decode_step ignores it. */
typedef struct {
  double tau;
  double eps;
  double rms_eps;
  int capacity;
  int score_mode;
  dla_dtype out_dtype;
  int from_cache;
  const int32_t* seq_lens;
} dla_params;

/* The state cache M of Algorithm 2 for B x H streams (device memory, caller
 * owned).  Physical slots hold the states; `slot` maps logical order (0 =
 * oldest) to physical slots so that merges move no state data.
 *   states [B][H][C][d_v][d_k] fp32   physical slots
 *   slot   [B][H][C] int32           logical -> physical (a permutation of
 *                                    0..m-1 on the first m entries)
 *   n      [B][H][C] int32           tokens per state, logical order
 *   ibar   [B][H][C] double          summed token scores, logical order
 *   m      [B][H]    int32           live states (including the open one) */
typedef struct {
  float* states;
  int32_t* slot;
  int32_t* n;
  double* ibar;
  int32_t* m;
  int B, H, C, dk, dv;
} dla_cache;

/* Fills *p with the defaults listed above. */
void dla_default_params(dla_params* p);

/* Bytes of one contiguous device block that dla_cache_carve can split into a
 * cache for B x H streams (256-byte aligned sub-arrays). */
size_t dla_cache_bytes(int B, int H, int C, int dk, int dv);

/* Points the members of *out into `base` (device memory of at least
 * dla_cache_bytes(...) bytes, 256-byte aligned).  Enqueues nothing. */
dla_status dla_cache_carve(void* base, size_t bytes, int B, int H, int C, int dk, int dv,
                           dla_cache* out);

/* Empties every stream's cache: m = 0, slot = identity, n = 0, ibar = 0
 * (Algorithm 2, "M <- [ ]").  State data is not cleared: slots >= m are never
 * read. */
dla_status dla_init_cache(const dla_cache* cache, void* stream);

/* Workspace bytes dla_forward needs for these sizes.  with_output = 0 sizes it
 * for a call with o == NULL (no read-out staging).  dla_forward accepts any
 * workspace at least dla_forward_min_workspace(...) large and splits the
 * sequence into more passes when it is smaller than this preferred size. */
size_t dla_forward_workspace(const dla_params* p, int B, int T, int H, int dk, int dv,
                             dla_dtype in_dtype, int with_output);
size_t dla_forward_min_workspace(const dla_params* p, int B, int T, int H, int dk, int dv,
                                 dla_dtype in_dtype, int with_output);

/* Waits for `stream` (a cudaStream_t) to complete its work, then returns the
 * device status of the library's calls enqueued on it since the previous
 * dla_sync_status on that stream, and clears it: DLA_OK, DLA_ERR_TIMEOUT (a
 * bounded device wait gave up) or DLA_ERR_DEVICE_CHECK (a kernel found an
 * inconsistent cache, snapshot list or pool); DLA_ERR_CUDA if the stream
 * could not be synchronised.  Each status word belongs to a (device, stream)
 * pair; a device keeps 255 of them for its first 255 streams and one shared
 * word for every later stream.  A stream handle that is destroyed and reused
 * inherits an unread status. */
dla_status dla_sync_status(void* stream);

/* Prefill / training-shaped forward over T tokens of B x H streams
 * (Algorithm 1 + Algorithm 2 + Eq. capacity_bounded_output).
 *   q, k, v, lam, o, boundary, merge_log: layouts above; o, lam, boundary and
 *   merge_log may be NULL (lam NULL = all ones; o NULL skips the read-out).
 *   cache: optional.  If given (dims B, H, C = p->capacity, d), it receives
 *   the final cache; with p->from_cache = 1 it is also the starting cache.
 *   With cache == NULL the cache lives in the workspace and from_cache must
 *   be 0.
 *   workspace: device memory of ws_bytes >= dla_forward_min_workspace(...).
 *   Its first 4 bytes receive the device status of the call once the work has
 *   run (int32: 0 ok, DLA_ERR_TIMEOUT when a bounded wait of a kernel gave up,
 *   DLA_ERR_DEVICE_CHECK when a kernel found an inconsistent cache or pool);
 *   the same status goes to the stream's status word (dla_sync_status).
 *   Schedule (bf16, d = 128, workspace of at least dla_forward_workspace(...)):
 *   the environment variable DLA_SCHEDULE, read at every call, selects
 *   "concurrent" (default: the scan runs once over the whole sequence while
 *   the Gram pre-pass and then the read-out run beside it on another stream,
 *   each waiting for the other side's progress; a kernel of the read-out side
 *   waits up to ~2 s for the scan to become resident, so the device should not
 *   be saturated by other work at that moment), "rounds" (the scan and the
 *   read-out alternate round by round on two internal streams) or "serial"
 *   (pre-pass, whole scan and read-out one after another, each kernel alone on
 *   the device: for timing and profiling).  The concurrent schedule needs
 *   every scan CTA resident at once with SMs to spare; calls with more streams
 *   than that take the rounds schedule.  All give the same results.
 *   DLA_SCAN (read at every call): unset selects the scan on warp-level tensor
 *   cores (CTA pairs, the open state in registers); "tc" selects, for calls
 *   with a read-out over whole rows of device-resident inputs, the scan on
 *   tcgen05 with the open state in tensor memory (one CTA per stream; same
 *   results, currently slower). */
dla_status dla_forward(const dla_params* p, dla_dtype in_dtype, int B, int T, int H, int dk,
                       int dv, const void* q, const void* k, const void* v, const float* lam,
                       void* o, const dla_cache* cache, uint8_t* boundary, int32_t* merge_log,
                       void* workspace, size_t ws_bytes, void* stream);

/* dla_forward over a packed batch of B rows of different lengths (ragged
 * batches without padding, as in serving; Sec. 3.2's fixed-size memory per
 * sequence makes each row an independent stream per head).  Row b holds tokens
 * cu_seqlens[b] .. cu_seqlens[b+1] - 1 of
 *   q, k, v   [total_tokens, H, d]   (bf16 or fp32)
 *   lam       [total_tokens, H, C]   fp32, or NULL (all ones)
 *   o         [total_tokens, H, d_v] (p->out_dtype), or NULL
 * and runs exactly as a call on its own tokens would (Algorithm 1 and 2 per
 * (row, head) stream, the read-out of Eq. capacity_bounded_output).
 *   cu_seqlens  device int32 [B + 1], 4-byte aligned: non-decreasing offsets
 *               with 0 <= cu_seqlens[b] and cu_seqlens[B] <= total_tokens.
 *   max_seqlen  an upper bound of every row's length; it takes the place of T
 *               in the workspace size (dla_forward_workspace(p, B, max_seqlen,
 *               ...)) and in the trace layout: boundary and merge_log are
 *               [B, H, max_seqlen], the row's tokens first, then padding
 *               (boundary 0, merge_log -1).
 *   cache       as in dla_forward ([B, H, C] streams, one per row and head).
 *   p->seq_lens must be NULL.  Offsets that break the rules above are found
 *   on the device: the row is clamped into range and the call's status is
 *   DLA_ERR_DEVICE_CHECK (dla_sync_status).  Inputs must be device-resident
 *   (there is no host-buffer variant).  DLA_SCAN=tc does not apply. */
dla_status dla_forward_varlen(const dla_params* p, dla_dtype in_dtype, int B, int max_seqlen,
                              long long total_tokens, const int32_t* cu_seqlens, int H, int dk, int dv,
                              const void* q, const void* k, const void* v, const float* lam, void* o,
                              const dla_cache* cache, uint8_t* boundary, int32_t* merge_log,
                              void* workspace, size_t ws_bytes, void* stream);

/* dla_forward for callers that cannot allocate device memory (the paper has
 * no counterpart: this is a deployment convenience).  Some callers cannot
 * call cudaMalloc where they run the forward pass -- for example a plugin of
 * an inference engine that owns all device memory and hands out no workspace,
 * or code running while another thread captures a CUDA graph in global mode,
 * where an allocation is an error.  This entry point takes the same arguments
 * as dla_forward minus the workspace: its scratch is a static device array of
 * 64 MiB compiled into the library, which every GPU that loads the library
 * holds until the process exits.  It allocates nothing.
 *   - The first call on each device (with that device current) looks up the
 *     array's device address with cudaGetSymbolAddress, and the first call
 *     from each host thread creates that thread's internal streams and events
 *     (as for dla_forward); make those first calls before any stream capture.
 *   - A call whose workspace need exceeds 64 MiB returns DLA_ERR_WORKSPACE with
 *     a message naming the limit; pass your own `cache` (and boundary /
 *     merge_log arrays) to keep the need small, or use dla_forward.
 *   - Every call shares the one array and rewrites the parts it reads; calls
 *     that overlap on the GPU (different streams, or different host threads,
 *     on the same device) race on it and must be serialised by the caller.
 *   - The call's device status (a bounded wait that gave up, a failed device
 *     check) goes to its stream's status word: read it with
 *     dla_sync_status(stream). */
dla_status dla_forward_noalloc(const dla_params* p, dla_dtype in_dtype, int B, int T, int H,
                               int dk, int dv, const void* q, const void* k, const void* v,
                               const float* lam, void* o, const dla_cache* cache,
                               uint8_t* boundary, int32_t* merge_log, void* stream);

/* Workspace bytes dla_forward_host needs for these sizes: device buffers for
 * q, k, v, lambda and o plus dla_forward_workspace(...).  0 for bad arguments. */
size_t dla_forward_host_workspace(const dla_params* p, int B, int T, int H, int dk, int dv,
                                  dla_dtype in_dtype, int with_output);

/* dla_forward with q, k, v, lam and o in HOST memory (same layouts and
 * semantics; the paper has no counterpart: this is the end-to-end call of a
 * caller whose tensors live on the host).  Whole rows only: p->seq_lens must
 * be NULL (DLA_ERR_UNSUPPORTED otherwise; ragged rows take dla_forward with
 * device-resident inputs, since the copies move whole rows and the o rows
 * past a row's length could not stay unwritten).  Page-locked host memory
 * (cudaHostAlloc / cudaHostRegister) makes the copies asynchronous; with
 * pageable memory they still work but do not overlap anything.
 *   cache, boundary, merge_log: device memory, as in dla_forward.
 *   workspace: device memory of ws_bytes >= dla_forward_host_workspace(...)
 *   (256-byte aligned); the input and output buffers are carved from its end,
 *   the rest is dla_forward's workspace (its status word first).
 * On the concurrent schedule (see dla_forward) the inputs are copied in 16
 * pieces of whole 64-token chunks on an internal stream, each piece followed
 * by a stream memory write of the count of pieces in place; the scan waits
 * (bounded) for the piece of every chunk it loads and forms its Gram entries
 * itself, the read-out follows the scan, and o goes back in 16 pieces on
 * another internal stream, each after a stream wait for the count of its
 * read-out CTAs, so the copies overlap the work.  On the other schedules the
 * inputs are copied first and o after the read-out.  The call only enqueues work: the host buffers
 * must stay valid, and o is filled, once `stream` has completed it.  Results
 * equal dla_forward's on the same inputs (decisions bit-identical; the
 * outputs to rounding of the Gram sums). */
dla_status dla_forward_host(const dla_params* p, dla_dtype in_dtype, int B, int T, int H, int dk,
                            int dv, const void* q, const void* k, const void* v, const float* lam,
                            void* o, const dla_cache* cache, uint8_t* boundary, int32_t* merge_log,
                            void* workspace, size_t ws_bytes, void* stream);

/* One recurrent step (Sec. 3.1 inference rule + Algorithm 2 + read-out) for
 * every stream: token (q, k, v) [B, H, d] against the persistent cache, which
 * is updated in place.  lam [B, H, C] fp32 or NULL; o [B, H, d] (out_dtype);
 * boundary [B, H] uint8 or NULL; merge_idx [B, H] int32 (i* or -1) or NULL.
 * p->capacity must equal cache->C.  A cache whose live count or slot map is
 * out of range is clamped and reported as DLA_ERR_DEVICE_CHECK through the
 * stream's status word (dla_sync_status). */
dla_status dla_decode_step(const dla_params* p, const dla_cache* cache, dla_dtype in_dtype,
                           const void* q, const void* k, const void* v, const float* lam,
                           void* o, uint8_t* boundary, int32_t* merge_idx, void* stream);

/* Gradients of the read-out with the forward pass's decisions held fixed
 * (training-shaped sequences).  The boundary and merge decisions of Algorithm 1
 * and 2 are piecewise constant in k and v, so their derivative is zero almost
 * everywhere; with them fixed, every state is a sum of token states over a
 * contiguous token range and Eq. capacity_bounded_output reads
 *   o_t = sum_{s <= t} lambda_{t, slot_t(s)} (q_t . k_s) v_s,
 * slot_t(s) the logical slot of the state holding token s after token t.  For
 * a loss L with grad_o = dL/do this call writes
 *   grad_q, grad_k, grad_v [B, T, H, d] fp32 and grad_lam [B, T, H, C] fp32
 *   (NULL: not computed; 0 for slots >= m_t),
 * taking q, k, v [B, T, H, d] (bf16 only: DLA_ERR_UNSUPPORTED otherwise), lam
 * [B, T, H, C] fp32 or NULL (all ones), grad_o [B, T, H, d] fp32 and the
 * decision trace of the forward call on the same inputs (boundary [B, H, T]
 * uint8, merge_log [B, H, T] int32).  p->capacity is the C of lam and of the
 * trace; p->from_cache must be 0 (the sequence starts from an empty cache) and
 * p->seq_lens NULL.  The work is quadratic in T per stream (every token pair).
 * A trace that is not a valid replay of Algorithm 2 (a merge index outside the
 * live pairs, a boundary into a full cache without a merge) is reported as
 * DLA_ERR_DEVICE_CHECK through the stream's status word; the gradients are
 * then undefined.  workspace: device memory of at least
 * dla_backward_workspace(...) bytes, 256-byte aligned; its first 4 bytes
 * receive the call's device status.  All pointers 16-byte aligned (lam and
 * grad_lam 4-byte). */
size_t dla_backward_workspace(const dla_params* p, int B, int T, int H, int dk, int dv, dla_dtype in_dtype);
dla_status dla_backward(const dla_params* p, dla_dtype in_dtype, int B, int T, int H, int dk, int dv,
                        const void* q, const void* k, const void* v, const float* lam,
                        const uint8_t* boundary, const int32_t* merge_log, const float* grad_o,
                        float* grad_q, float* grad_k, float* grad_v, float* grad_lam,
                        void* workspace, size_t ws_bytes, void* stream);

/* Instrumentation (no counterpart in the paper).  Kernel kinds of the
 * library: K1 scan, K2 read-out, K3 decode, cache init, K0 Gram pre-pass, the
 * one-thread gate of the concurrent schedule, the one-thread kernel that
 * folds a call's status into its stream's status word, and K4 (the three
 * kernels of dla_backward). */
typedef enum {
  DLA_K_SCAN = 0,
  DLA_K_READOUT = 1,
  DLA_K_DECODE = 2,
  DLA_K_INIT = 3,
  DLA_K_GRAM = 4,
  DLA_K_GATE = 5,
  DLA_K_STATUS = 6,
  DLA_K_BACKWARD = 7,
  DLA_K_COUNT = 8
} dla_kernel_kind;

/* enable = 1: from now on, every kernel this host thread launches through the
 * library is bracketed by two CUDA events recorded on its stream (a few
 * microseconds of host overhead per launch, none on the device).  enable = 0
 * stops recording.  Returns DLA_ERR_CUDA if events cannot be created. */
dla_status dla_timing_enable(int enable);

/* Waits for the recorded events, then writes per kernel kind the number of
 * launches (launches[DLA_K_COUNT], host memory) and their summed device time in
 * milliseconds (ms[DLA_K_COUNT]).  reset = 1 forgets the records afterwards. */
dla_status dla_timing_read(int* launches, double* ms, int reset);

/* Message of the last error returned on this host thread ("" if none). */
const char* dla_last_error(void);

/* Short name of a status code. */
const char* dla_status_string(dla_status s);

/* DLA_VERSION of the built library. */
int dla_version(void);

#ifdef __cplusplus
}
#endif

#endif /* DLA_H */
