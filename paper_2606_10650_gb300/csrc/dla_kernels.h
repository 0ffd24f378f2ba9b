// dla_kernels.h -- internal launch interface between the C ABI (dla_api.cu)
// and the kernels.  Not part of the public header.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "dla.h"

namespace dla {

constexpr int kMaxC = 64;   // largest capacity C with the capacity merge of Algorithm 2 on the GPU
// Largest C of the DLA(I) instances (Table 5: dynamic merging only): bf16
// inputs, d = 128, capacities above kMaxC hold up to kMaxCBig states without
// merge machinery; a stream that would need a capacity merge fails the call's
// device check.
constexpr int kMaxCBig = 256;
constexpr int kScanL = 64;  // tokens per scan chunk (K1)
// Floats per chunk of the Gram pre-pass output: suffix table gs[j][t], its
// prefix table Q[j][t], a_t, and the exclusive prefix sums
// SA[t] = sum_{u < t} sqrt(a_u) for t = 0 .. 64 (|v_u| |k_u| = sqrt(a_u): the
// growth of a state's norm bound), padded to a multiple of four (see GramArgs).
constexpr int kGramSA = 2 * kScanL * kScanL + kScanL;
constexpr int kGramBlock = kGramSA + kScanL + 4;

// Gram block of the tensor-core scan (K0 with GramArgs::packed = 1), per chunk:
//   gs[j][t], j <= t <= 64   packed by rows (row j starts at 65 j - j (j - 1) / 2)
//   Q[j][t],  j <= t <= 64   the same packing (Q[j][64] is the whole chunk's running sum)
//   a[t]                     64
//   cs[j][t] = sum_{j <= s < 64} (k_t.k'_s)(v_t.v'_s), t in this chunk, s in the
//            previous chunk (k', v'): beta_t of a segment opened at j of the
//            previous chunk, 64 x 64 row-major
constexpr int kPackTri = 65 * kScanL - kScanL * (kScanL - 1) / 2;  // 2144
constexpr int kGramBlockTc = 2 * kPackTri + kScanL + kScanL * kScanL;
__host__ __device__ constexpr int pack_row(int j) { return 65 * j - j * (j - 1) / 2; }
// Floats between consecutive chunks' blocks in the Gram pre-pass output (either
// layout).
constexpr int kGramStride = kGramBlockTc;
static_assert(kGramStride >= kGramBlock && (kGramBlock * 4) % 16 == 0, "Gram block layout");

// Method parameters of the score / boundary test (Sec. 3.1).
struct ScoreParams {
  double tau, eps, rms_eps;
  int score_mode;
  // fp32 copies: tau_f is the smallest float >= tau, so that for a float score
  // I >= tau_f exactly when (double) I >= tau; eps_f, rms_eps_f rounded to nearest
  float tau_f, eps_f, rms_eps_f;
};

// Fills the fp32 fields of sp from its fp64 ones (host).
void finish_score_params(ScoreParams& sp);

// K1: sequential scan of one round [t_begin, t_end) of every stream.
struct ScanArgs {
  const void* k;
  const void* v;
  int B, T, H;
  int t_begin, t_end;
  ScoreParams sp;
  int C;
  // live cache (fp32 states in physical slots, logical metadata)
  float* states;
  int32_t* slot;
  int32_t* n;
  double* ibar;
  int32_t* m;
  // per-token trace [B, H, T]
  uint8_t* boundary;
  int32_t* merge_log;
  // read-out snapshots (pool == nullptr: no read-out in this call)
  void* pool;
  int pool_cap;          // entries per stream
  int32_t* snap_m0;      // [B*H][snap_stride]     live entries at each interval start
  int32_t* snap_ids;     // [B*H][snap_stride][C]  their pool ids (logical order)
  int snap_stride;       // intervals of the whole sequence
  int snap_base;         // global index of this round's first interval
  int nsnap;             // snapshot intervals in this round
  int snap_chunks;       // scan chunks per snapshot interval
  int carry_in;          // 1: the pool continues from the previous round (pstate holds its counters)
  int snap_at_end;       // 1: also snapshot at this round's last interval end (for the next round)
  int32_t* pstate;       // [B*H] next free pool entry, then [B*H][C] pool ids of the live entries
  // fp16 pool (tensor-core read-out): the scale s of each entry (S / s is stored),
  // [B*H][pool_cap], and upper bounds of the live entries' norms |S|_F, [B*H][C]
  // (read at a round's start, written at its end; a call continuing from a
  // cache gets them from launch_cache_bounds first)
  float* pool_scale;
  float* nbound;
  const float* gram;     // Gram pre-pass output [B*H][gram_chunks][kGramBlock], or nullptr
  int gram_chunks;       // 64-token chunks of the whole sequence
  // Gram pre-pass running beside the scan (nullptr: it finished before the
  // scan started; the pre-pass then starts at chunk 0): [B*H][gram_nblk] chunks
  // written so far by the pre-pass CTA of each block (block b: chunks b,
  // b + gram_nblk, ..., written in that order)
  const int32_t* gram_ready;
  int gram_nblk;
  // Inputs streamed in by the host (nullptr: resident before the launch): the
  // count of pieces of piece_chunks 64-token chunks whose k, v (and q, lambda)
  // rows have arrived, written in stream order after each piece's copies
  const int32_t* piece_ready;
  int piece_chunks;
  const int32_t* seq_lens;  // [B] tokens of each row (padding after them), or nullptr: T each
  // [B] token row of each batch row's first token (the packed layout: rows of
  // seq_lens[b] tokens one after another), or nullptr: b * T (the padded layout).
  // Set only together with seq_lens.
  const int32_t* row_start;
  int32_t* progress;     // [B*H][2] intervals completed by each CTA of the stream, or nullptr
  int32_t* started;      // counter of the scan CTAs that have started, or nullptr
  int32_t* status;       // device status word (0 = ok)
};

// K0: Gram pre-pass over every 64-token chunk of every stream (bf16 inputs).
// Per chunk, with G_ts = (k_t.k_s)(v_t.v_s):
//   gs[j][t] = sum_{j <= s < t} G_ts       (beta_t of a segment opened at j, without S)
//   Q[j][t]  = sum_{j <= u < t} gs[j][u]   (their running sum over the segment)
//   a_t      = G_tt
// One CTA per (stream, block): block b of a launch takes its chunks chunk0 + b,
// chunk0 + b + nblk, ... in order, loading the next while it computes this one.
struct GramArgs {
  const void* k;
  const void* v;
  int B, T, H;
  int nchunks;           // chunks of the whole sequence
  int chunk0, count;     // this launch: chunks chunk0 .. chunk0 + count - 1
  int nblk, per_blk;     // blocks of this launch and chunks per block at most (nblk * per_blk >= count)
  float* out;            // [B*H][nchunks][kGramBlock]: gs (64 x 64), Q (64 x 64), a (64); packed: [kGramBlockTc]
  int32_t* ready;        // [B*H][nblk] chunks of the block written so far (published after its first four, then every fourth), or nullptr
  int packed;            // 1: the tensor-core scan's layout (kGramBlockTc floats per chunk, with the cross table)
  // per-row lengths and first token rows (as in ScanArgs), or nullptr: rows of T
  // tokens at b * T.  Rows past a row's length are zero-filled, not read.
  const int32_t* seq_lens;
  const int32_t* row_start;
};
constexpr int kMaxGramBlk = 64;  // blocks per stream of one Gram launch, at most
constexpr int kGramCtasPerSm = 3;  // resident Gram CTAs per SM (shared memory)
constexpr int kGramTcCtasPerSm = 2;  // the same for the packed layout (two chunks of k, v in shared memory)

// K2: read-out of one round, one CTA per (snapshot interval, stream).
struct ReadoutArgs {
  const void* q;
  const void* k;
  const void* v;
  const float* lam;      // [B, T, H, C] or nullptr
  void* o;               // [B, T, H, d]
  int out_bf16;
  int B, T, H, C;
  int t_begin, t_end;
  const uint8_t* boundary;
  const int32_t* merge_log;
  const void* pool;
  const float* pool_scale;  // fp16 pool: the scale of each entry ([B*H][pool_cap])
  int pool_cap;
  const int32_t* snap_m0;
  const int32_t* snap_ids;
  int snap_stride;       // intervals of the whole sequence
  int snap_base;         // global index of this round's first interval
  int nsnap;
  int interval;          // tokens per snapshot interval
  const int32_t* progress;  // [B*H][2] scan progress to wait for (the scan runs concurrently), or nullptr
  int progress_ctas;        // scan CTAs per stream (1 or 2): entries of progress[bh] that count
  // Output copied back piece by piece while the read-out runs (tensor-core
  // read-out), or nullptr: every CTA (one per interval and stream) adds 1 to
  // out_done[(interval / 2) / out_piece_pairs] once its rows of o are stored
  // (after a device-scope fence)
  int32_t* out_done;
  int out_piece_pairs;
  const int32_t* seq_lens;  // [B] tokens of each row (padding after them), or nullptr: T each
  const int32_t* row_start; // [B] first token row of each batch row (packed layout), or nullptr: b * T
  long long total_rows;     // token rows of q, k, v, lambda and o in the packed layout (row_start set)
  int lam_l2;  // 1: lambda arrives while the kernel runs (streamed inputs): read it through L2
  int32_t* status;          // device status word
};

// K3: one decode step of every stream.
struct DecodeArgs {
  const void* q;
  const void* k;
  const void* v;
  const float* lam;      // [B, H, C] or nullptr
  void* o;               // [B, H, d]
  int out_bf16;
  int B, H, C;
  ScoreParams sp;
  float* states;
  int32_t* slot;
  int32_t* n;
  double* ibar;
  int32_t* m;
  uint8_t* boundary;     // [B, H] or nullptr
  int32_t* merge_idx;    // [B, H] or nullptr
  int32_t* status;       // device status word of the call's stream (6 when the cache is inconsistent)
};

// K4: gradients of the read-out with the forward pass's decisions held fixed
// (dla_backward.cu).  bf16 q, k, v [B, T, H, d]; fp32 g = dL/do and gradients.
struct BackwardArgs {
  const void* q;
  const void* k;
  const void* v;
  const float* lam;          // [B, T, H, C] or nullptr (ones)
  const float* g;            // [B, T, H, d]
  const uint8_t* boundary;   // [B, H, T] of the forward pass
  const int32_t* merge_log;  // [B, H, T]
  float* dq;
  float* dk;
  float* dv;
  float* dlam;               // [B, T, H, C] or nullptr
  int B, T, H, C;
  int32_t* evt;              // workspace: [B*H][T] boundary events at or before each token
  int32_t* firsts;           // workspace: [B*H][T + 1][kMaxC] first tokens of the live states after each event
  int32_t* status;           // device status word (6: an inconsistent trace)
};
// The three kernels of K4, in this order on one stream: the slot lists, then
// dK and dV, then dQ and dlambda.
cudaError_t launch_backward_slots(const BackwardArgs& a, cudaStream_t s);
cudaError_t launch_backward_dkv(const BackwardArgs& a, int d, cudaStream_t s);
cudaError_t launch_backward_dq(const BackwardArgs& a, int d, cudaStream_t s);
// Workspace bytes of the slot lists of launch_backward.
size_t backward_slot_bytes(int BH, int T);

// Norms |S_i|_F of the live states of a cache (logical order, i < m), rounded
// up, into out[B*H][C]: the norm bounds a forward call that continues from the
// cache starts with.
cudaError_t launch_cache_bounds(const float* states, const int32_t* slot, const int32_t* m, int BH, int C, int d,
                                float* out, cudaStream_t s);

// Per-row lengths and first token rows of a packed batch from its cumulative
// offsets cu[0..B] (device int32): lens[b] = cu[b+1] - cu[b] and start[b] = cu[b],
// checked (0 <= cu[b] <= cu[b+1] <= total, length <= T); a row that fails the
// check sets status 6 and is clamped into range, so no kernel reads outside
// the total rows.
cudaError_t launch_varlen_rows(const int32_t* cu, int B, int T, long long total, int32_t* lens, int32_t* start,
                               int32_t* status, cudaStream_t s);

// Records a formatted message as the calling thread's dla_last_error() and
// returns s (for entry points defined outside dla_api.cu).
dla_status set_error(dla_status s, const char* fmt, ...);

// K1 on CUDA cores for fp32 inputs (dla_scan.cu), fp32 pool entries.
cudaError_t launch_scan(const ScanArgs& a, int d, cudaStream_t s);
// K1 for bf16 inputs with its contractions on mma.sync (dla_scan_mma.cu).
cudaError_t launch_scan_mma(const ScanArgs& a, int d, bool pool_f16, cudaStream_t s);
// CTAs per stream of launch_scan_mma: 2 (a CTA pair) when 2*B*H CTAs fit the
// device's SMs in one wave with d = 128, else 1.
int scan_mma_ctas_per_stream(int BH, int d);
// Streams whose launch_scan_mma CTAs (pairs or single CTAs, as
// scan_mma_ctas_per_stream picks for BH streams) can all be resident at once.
int scan_mma_resident_streams(int BH, int d);
// Block count of a Gram launch over `count` chunks of BH streams whose CTAs
// fit `slots` resident CTAs (kGramCtasPerSm per SM) in one wave (at least one block per
// stream, at most kMaxGramBlk); per_blk follows.
void gram_blocks(int BH, int count, int slots, int* nblk, int* per_blk);
// One CTA that returns once `n` scan CTAs have started (*started >= n), or after
// ~2 s with status 5: the read-out stream runs it before its first launch, so
// that read-out CTAs waiting for the scan never hold the SMs the scan needs.
cudaError_t launch_gate(const int32_t* started, int n, int32_t* status, cudaStream_t s);
// Loads the code of the kernels of the concurrent scan / read-out path on the
// current device (cudaFuncGetAttributes).  With lazy module loading, a kernel's
// first launch can wait for the device's running kernels, and a read-out
// waiting for a scan whose code is not loaded yet would wait until its time
// limit: the forward pass calls these before its first launch.
cudaError_t preload_scan_kernels();
cudaError_t preload_readout_kernels();
cudaError_t launch_gram(const GramArgs& a, int d, cudaStream_t s);
// K1 on tcgen05 (dla_scan_tc.cu): bf16 inputs, d = 128, one CTA per stream, the
// open state in tensor memory; needs the packed Gram pre-pass output, whole rows
// (no per-row lengths) and resident inputs.
cudaError_t launch_scan_tc(const ScanArgs& a, cudaStream_t s);
// Streams whose launch_scan_tc CTAs can all be resident at once.
int scan_tc_resident_streams();
cudaError_t preload_scan_tc_kernel();
size_t scan_smem_bytes(int d);
cudaError_t launch_readout_simt(const ReadoutArgs& a, int d, bool in_bf16, cudaStream_t s);
constexpr int kReadoutSimtInterval = 64;
// K2 for bf16 inputs, d = 128, 128-token intervals (tcgen05 / TMEM / TMA,
// snapshots stored as bf16 hi + lo): one CTA per pair of intervals computes the
// snapshot part and the intra-interval part and writes o.
cudaError_t launch_readout_tc(const ReadoutArgs& a, int32_t* status, cudaStream_t s);
constexpr int kReadoutTcInterval = 128;
cudaError_t launch_decode(const DecodeArgs& a, int d, bool in_bf16, cudaStream_t s);
cudaError_t launch_init_cache(int32_t* slot, int32_t* n, double* ibar, int32_t* m, int BH, int C,
                              cudaStream_t s);

}  // namespace dla
