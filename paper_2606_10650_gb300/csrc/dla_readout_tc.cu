// dla_readout_tc.cu -- K2b on the 5th-generation tensor cores (tcgen05 + TMEM
// + TMA): the snapshot part of the read-out of Eq. (capacity_bounded_output)
//   o_t = o_intra[t] + sum_{x < m0} lambda_{t, L_t(x)} (S_x q_t)
// for one 128-token interval of one stream per CTA, bf16 inputs, d = 128.
// o_intra (the interval's own tokens, fp32) comes from K2a.  The cache seen by
// token t is the snapshot taken by K1 at the interval start (m0 states,
// logical order) regrouped by the merges decided inside the interval: merges
// only add states, so snapshot entry x contributes with the lambda of its
// logical slot L_t(x) after the interval's events up to t.
// Per state x: D_x = Q S_x^T = Q (S_hi + S_lo)^T (M = 128 tokens, N = 128,
// K = 128), the fp32 snapshot split into bf16 hi + lo parts by K1 (two MMAs per
// state keep the state rounding near 2^-17 instead of 2^-9).
// Roles: warp 0 issues TMA loads into five 32 KB half-stages (the hi or lo part
// of one state each), warp 1 issues tcgen05.mma (one thread) into four TMEM
// accumulators of 128 columns, warps 2..9 read TMEM, weight by lambda and
// accumulate o in registers (warp w reads TMEM lane quadrant w % 4; warps 2-5
// own columns 0-63, warps 6-9 own 64-127).
#include <cudaTypedefs.h>

#include "dla_common.cuh"
#include "dla_sm100.cuh"

namespace dla {

namespace {

using namespace sm100;

constexpr int L = 128;   // tokens per CTA
constexpr int D = 128;   // head dimension
constexpr int NT = 320;  // 10 warps
constexpr int NEPI = 8;  // epilogue warps
constexpr int NHS = 5;   // shared-memory half-stages
constexpr int NACC = 4;  // TMEM accumulators
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTile = L * 128;  // one K-major 128B-swizzled tile: 128 rows x 64 bf16

struct TcSmem {
  uint8_t Q[2][kTile];                 // A operand, two k-halves              32 KB
  uint8_t hs[NHS][2][kTile];           // [half-stage][k-half]                160 KB
  unsigned char tab[(L + 1) * kMaxC];  // L(x) of snapshot entry x after event e
  int logi[kMaxC];
  int evt[L];                          // events (boundaries) at or before token t
  int mlog[L];                         // the interval's merge indices
  uint8_t bnd[L];                      // and boundary flags
  int ids[kMaxC];                      // pool ids of the snapshot entries
  uint64_t bar_q, bar_done;
  uint64_t full[NHS], empty[NHS], acc_full[NACC], acc_empty[NACC];
  uint32_t tmem_base;
  int abort_flag;
};

}  // namespace

__global__ void __launch_bounds__(NT, 1)
    readout_tc_kernel(ReadoutArgs a, const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmS,
                      int32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  TcSmem& sm = *reinterpret_cast<TcSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int s = blockIdx.x, bh = blockIdx.y;
  const int b = bh / a.H, h = bh % a.H;
  const int C = a.C;
  const int c0 = a.t_begin + s * L;
  const int Lc = min(L, a.t_end - c0);
  const long long lrow = (long long)bh * a.snap_stride + a.snap_base + s;
  const int m0 = a.snap_m0[lrow];
  volatile int* abort = &sm.abort_flag;

  if (tid == 0) {
    mbar_init(&sm.bar_q, 1);
    mbar_init(&sm.bar_done, 1);
    for (int i = 0; i < NHS; ++i) {
      mbar_init(&sm.full[i], 1);
      mbar_init(&sm.empty[i], 1);
    }
    for (int i = 0; i < NACC; ++i) {
      mbar_init(&sm.acc_full[i], 1);
      mbar_init(&sm.acc_empty[i], NEPI);
    }
    sm.abort_flag = 0;
    fence_mbar_init();
  }
  for (int i = tid; i < m0; i += NT) sm.ids[i] = a.snap_ids[lrow * C + i];
  if (warp == 1) tmem_alloc(&sm.tmem_base, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      prefetch_tmap(&tmQ);
      prefetch_tmap(&tmS);
      mbar_expect_tx(&sm.bar_q, 2 * kTile);
      tma_load_4d(sm.Q[0], &tmQ, &sm.bar_q, 0, h, c0, b);
      tma_load_4d(sm.Q[1], &tmQ, &sm.bar_q, 64, h, c0, b);
      int issued[NHS];  // uses of each half-stage so far
      for (int i = 0; i < NHS; ++i) issued[i] = 0;
      for (int u = 0; u < 2 * m0; ++u) {  // unit u: part u & 1 (hi, lo) of state u >> 1
        const int hsi = u % NHS, k = u / NHS;
        if (!mbar_wait(&sm.empty[hsi], (uint32_t)((k & 1) ^ 1), abort, status)) break;
        mbar_expect_tx(&sm.full[hsi], 2 * kTile);
        const int row = (int)((((long long)bh * a.pool_cap + sm.ids[u >> 1]) * 2 + (u & 1)) * D);
        tma_load_2d(sm.hs[hsi][0], &tmS, &sm.full[hsi], 0, row);
        tma_load_2d(sm.hs[hsi][1], &tmS, &sm.full[hsi], 64, row);
        issued[hsi] = k + 1;
      }
      if (*abort) {  // let copies in flight land before the CTA exits
        for (int i = 0; i < NHS; ++i)
          if (issued[i] > 0) mbar_wait(&sm.full[i], (uint32_t)((issued[i] - 1) & 1), abort, nullptr);
        mbar_wait(&sm.bar_q, 0, abort, nullptr);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(L, D);
      bool ok = mbar_wait(&sm.bar_q, 0, abort, status);
      for (int x = 0; ok && x < m0; ++x) {
        const int buf = x % NACC, kb = x / NACC;
        if (!mbar_wait(&sm.acc_empty[buf], (uint32_t)((kb & 1) ^ 1), abort, status)) break;
        tc_fence_after();
        const uint32_t dcol = tmem + 128u * buf;
        for (int part = 0; part < 2; ++part) {
          const int u = 2 * x + part, hsi = u % NHS, k = u / NHS;
          if (!(ok = mbar_wait(&sm.full[hsi], (uint32_t)(k & 1), abort, status))) break;
          tc_fence_after();
          for (int kk = 0; kk < 8; ++kk) {
            const uint32_t off = (uint32_t)(kk & 3) * 32;
            mma_bf16(dcol, desc_kmajor_sw128(smem_u32(sm.Q[kk >> 2]) + off),
                     desc_kmajor_sw128(smem_u32(sm.hs[hsi][kk >> 2]) + off), idesc, (part | kk) > 0);
          }
          mma_commit(&sm.empty[hsi]);
        }
        if (ok) mma_commit(&sm.acc_full[buf]);
      }
      mma_commit(&sm.bar_done);  // every MMA issued above has completed once this fires
      mbar_wait(&sm.bar_done, 0, abort, nullptr);
    }
  } else {
    // ------------------------------------------------------------ epilogue warps
    const int ew = warp - 2;            // 0..7
    const int quad = warp & 3;          // TMEM lane quadrant of this warp
    const int ch = (warp < 6) ? 0 : 1;  // column half
    const int t = quad * 32 + lane;     // token row of this thread
    const uint32_t lane_addr = tmem + ((uint32_t)(quad * 32) << 16);
    const int etid = ew * 32 + lane;    // 0..255
    const long long rowbase = ((long long)b * a.T + c0) * a.H + h;  // row index of token c0

    if (etid < L) {  // the interval's boundary flags and merge indices, staged once
      const bool in = etid < Lc;
      sm.bnd[etid] = in ? a.boundary[(long long)bh * a.T + c0 + etid] : (uint8_t)0;
      sm.mlog[etid] = in ? a.merge_log[(long long)bh * a.T + c0 + etid] : -1;
    }
    // o starts from the intra-interval part (K2a; column-quad order, so a warp
    // reads 512 contiguous bytes per load)
    float o[64];
    {
      const float* src = a.ointra + ((long long)bh * a.ointra_T + (c0 - a.t_begin)) * D + (16 * ch * L + t) * 4;
#pragma unroll
      for (int i = 0; i < 64; i += 4) {
        float4 v4 = make_float4(0.f, 0.f, 0.f, 0.f);
        if (t < Lc) v4 = *reinterpret_cast<const float4*>(src + (i / 4) * L * 4);
        o[i] = v4.x; o[i + 1] = v4.y; o[i + 2] = v4.z; o[i + 3] = v4.w;
      }
    }
    asm volatile("bar.sync 1, 256;" ::: "memory");
    // logical slots of the snapshot entries, one table row per boundary event
    // (one warp): row e holds L(x) after the first e events of the interval
    if (ew == 0) {
      for (int x = lane; x < m0; x += 32) {
        sm.logi[x] = x;
        sm.tab[x] = (unsigned char)x;
      }
      __syncwarp();
      unsigned long long lo64 = 0, hi64 = 0;
#pragma unroll
      for (int w4 = 0; w4 < 4; ++w4) {
        const unsigned m = __ballot_sync(0xffffffffu, sm.bnd[32 * w4 + lane] != 0);
        if (w4 < 2) lo64 |= (unsigned long long)m << (32 * w4);
        else hi64 |= (unsigned long long)m << (32 * (w4 - 2));
      }
      int ev = 0;
      while (lo64 | hi64) {
        const int tt = lo64 ? (__ffsll((long long)lo64) - 1) : (64 + __ffsll((long long)hi64) - 1);
        if (lo64) lo64 &= lo64 - 1; else hi64 &= hi64 - 1;
        const int j = sm.mlog[tt];
        ev += 1;
        for (int x = lane; x < m0; x += 32) {
          int li = sm.logi[x];
          if (j >= 0 && li > j) sm.logi[x] = --li;
          sm.tab[ev * kMaxC + x] = (unsigned char)li;
        }
      }
    }
    if (etid < L) {  // events at or before each token (warps 2..5, one token per lane)
      const int tt = etid;
      int e = 0;
#pragma unroll
      for (int w4 = 0; w4 < 4; ++w4) {
        const unsigned m = __ballot_sync(0xffffffffu, sm.bnd[32 * w4 + lane] != 0);
        if (32 * w4 + 31 <= tt) e += __popc(m);
        else if (32 * w4 <= tt) e += __popc(m & (0xffffffffu >> (31 - (tt - 32 * w4))));
      }
      sm.evt[tt] = e;
    }
    asm volatile("bar.sync 1, 256;" ::: "memory");
    const float* lam_t = (a.lam && t < Lc) ? a.lam + (rowbase + (long long)t * a.H) * C : nullptr;
    const unsigned char* tab_t = sm.tab + sm.evt[t] * kMaxC;
    // weight of state x for this token; fetched one state ahead of its use
    auto weight = [&](int x) -> float {
      if (t >= Lc || x >= m0) return 0.f;
      return lam_t ? lam_t[tab_t[x]] : 1.f;
    };
    float w_next = weight(0);
    for (int x = 0; x < m0; ++x) {
      const int buf = x % NACC, kb = x / NACC;
      const float w = w_next;
      w_next = weight(x + 1);
      if (!mbar_wait(&sm.acc_full[buf], (uint32_t)(kb & 1), abort, status)) break;
      tc_fence_after();
      float dv[32];
      const uint32_t base = lane_addr + 128u * buf + 64 * ch;
      tmem_ld32(base, dv);
#pragma unroll
      for (int i = 0; i < 32; ++i) o[i] += w * dv[i];
      tmem_ld32(base + 32, dv);
#pragma unroll
      for (int i = 0; i < 32; ++i) o[32 + i] += w * dv[i];
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.acc_empty[buf]);
    }
    if (t < Lc && !*abort) {
      const long long orow = (rowbase + (long long)t * a.H) * D + 64 * ch;
      if (a.out_bf16) {
        __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(a.o) + orow;
#pragma unroll
        for (int i = 0; i < 64; i += 4) store4(out + i, make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]));
      } else {
        float* out = reinterpret_cast<float*>(a.o) + orow;
#pragma unroll
        for (int i = 0; i < 64; i += 4) store4(out + i, make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]));
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// ---------------------------------------------------------------- host side
namespace {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// [B, T, H, 128] bf16 rows of one stream: dims (k, h, t, b), box (64, 1, 128, 1).
bool map_tokens(CUtensorMap* m, const void* base, int B, int T, int H) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)H, (cuuint64_t)T, (cuuint64_t)B};
  cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)H * D * 2, (cuuint64_t)T * H * D * 2};
  cuuint32_t box[4] = {64, 1, (cuuint32_t)L, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Snapshot pool as rows of 128 bf16: box (64, 128).
bool map_pool(CUtensorMap* m, const void* base, long long rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)D * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)L};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cudaError_t launch_readout_tc(const ReadoutArgs& a, int32_t* status, cudaStream_t st) {
  CUtensorMap mq, ms;
  const long long rows = (long long)a.B * a.H * a.pool_cap * 2 * D;
  if (!map_tokens(&mq, a.q, a.B, a.T, a.H) || !map_pool(&ms, a.pool, rows)) return cudaErrorInvalidValue;
  const size_t smem = sizeof(TcSmem) + 1024;
  cudaError_t e = cudaFuncSetAttribute(readout_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(a.nsnap, a.B * a.H);
  readout_tc_kernel<<<grid, NT, smem, st>>>(a, mq, ms, status);
  return cudaGetLastError();
}

size_t readout_tc_smem_bytes() { return sizeof(TcSmem) + 1024; }

}  // namespace dla
