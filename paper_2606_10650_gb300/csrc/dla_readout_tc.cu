// dla_readout_tc.cu -- K2 on the 5th-generation tensor cores (tcgen05 + TMEM
// + TMA): the read-out o_t = sum_i lambda_{t,i} S_i q_t of
// Eq. (capacity_bounded_output) for one 128-token interval of one stream per
// CTA, bf16 inputs, d = 128.
//
// Decomposition (same as the CUDA-core K2): the cache seen by token t is the
// snapshot taken by K1 at the interval start (m0 states, logical order),
// regrouped by the merges decided inside the interval, plus the interval's own
// tokens, so
//   o_t = sum_{x < m0} lambda_{t, L_t(x)} (S_x q_t)
//       + sum_{s <= t} lambda_{t, L_t(e(s))} (q_t . k_s) v_s.
// Tensor-core work per CTA (M = 128 tokens, N = 128, K = 128):
//   P  = Q K^T                        -> TMEM cols [0, 128)
//   O  = Pt V   (Pt = P * weights, bf16, written back to shared memory) -> [128, 256)
//   D_x = Q S_x^T = Q (S_hi + S_lo)^T -> [256, 384) / [384, 512), one per state
// The fp32 snapshot is split into bf16 hi + lo parts by K1 (two MMAs per
// state), keeping the state rounding error near 2^-17 instead of 2^-9.
// Roles: warp 0 issues TMA loads, warp 1 issues tcgen05.mma (one thread),
// warps 2..9 read TMEM, apply lambda and accumulate o in registers (warp w
// reads TMEM lane quadrant w % 4; warps 2-5 own columns 0-63, warps 6-9 own
// 64-127).  Shared-memory stages hold one state's hi + lo (64 KB) each; during
// the intra-interval phase stage A holds K and V^T instead.
#include <cudaTypedefs.h>

#include "dla_common.cuh"
#include "dla_sm100.cuh"

namespace dla {

namespace {

using namespace sm100;

constexpr int L = 128;           // tokens per CTA
constexpr int D = 128;           // head dimension
constexpr int NT = 320;          // 10 warps
constexpr int NEPI = 8;          // epilogue warps
constexpr int MAXE = kMaxC + L;  // entries visible inside one interval
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t COL_P = 0, COL_O = 128, COL_S = 256;
constexpr uint32_t kTile = L * 128;  // one K-major 128B-swizzled tile: 128 rows x 64 bf16

struct TcSmem {
  uint8_t Q[2][kTile];         // A operand, two k-halves                      32 KB
  uint8_t st[2][2][2][kTile];  // [stage][hi/lo][k-half]; stage 0 = A, 1 = B  128 KB
  uint8_t Pt[2][kTile];        // lambda-weighted P, A operand [t][s]           32 KB
  unsigned char tab[(L + 1) * MAXE];  // logical slot of entry x after event e    24 KB
  int ent[L];                   // entry holding token s
  int evt[L];                   // events (boundaries) at or before token t
  uint8_t bnd[L];               // the interval's boundary flags
  int mlog[L];                  // and merge indices
  int ids[kMaxC];               // pool ids of the snapshot entries
  uint64_t bar_qk, bar_p, bar_pt, bar_o, bar_done;
  uint64_t full[2], empty[2], acc_full[2], acc_empty[2];
  uint32_t tmem_base;
  int abort_flag;
};

// The stage of state x: even states use stage B (free at once), odd ones
// stage A (free after the intra-interval MMAs, which read K and V^T there).
__device__ __forceinline__ int stage_of(int x) { return (x & 1) ? 0 : 1; }

}  // namespace

__global__ void __launch_bounds__(NT, 1)
    readout_tc_kernel(ReadoutArgs a, const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmS, int32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  TcSmem& sm = *reinterpret_cast<TcSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int s = blockIdx.x, bh = blockIdx.y;
  const int b = bh / a.H, h = bh % a.H;
  const int C = a.C;
  const int c0 = a.t_begin + s * L;
  const int Lc = min(L, a.t_end - c0);
  const int m0 = a.snap_m0[(long long)bh * a.snap_stride + a.snap_base + s];
  volatile int* abort = &sm.abort_flag;

  if (tid == 0) {
    mbar_init(&sm.bar_qk, 1);
    mbar_init(&sm.bar_p, 1);
    mbar_init(&sm.bar_pt, NEPI);
    mbar_init(&sm.bar_o, 1);
    mbar_init(&sm.bar_done, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sm.full[i], 1);
      mbar_init(&sm.empty[i], 1);
      mbar_init(&sm.acc_full[i], 1);
      mbar_init(&sm.acc_empty[i], NEPI);
    }
    sm.abort_flag = 0;
    fence_mbar_init();
  }
  for (int i = tid; i < m0; i += NT) sm.ids[i] = a.snap_ids[((long long)bh * a.snap_stride + a.snap_base + s) * C + i];
  if (warp == 1) tmem_alloc(&sm.tmem_base, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      prefetch_tmap(&tmQ);
      prefetch_tmap(&tmK);
      prefetch_tmap(&tmS);
      mbar_expect_tx(&sm.bar_qk, 4 * kTile);
      tma_load_4d(sm.Q[0], &tmQ, &sm.bar_qk, 0, h, c0, b);
      tma_load_4d(sm.Q[1], &tmQ, &sm.bar_qk, 64, h, c0, b);
      tma_load_4d(sm.st[0][0][0], &tmK, &sm.bar_qk, 0, h, c0, b);
      tma_load_4d(sm.st[0][0][1], &tmK, &sm.bar_qk, 64, h, c0, b);
      int issued[2] = {0, 0};
      for (int x = 0; x < m0; ++x) {
        const int st = stage_of(x), k = x >> 1;
        const uint32_t par = (st == 0) ? (uint32_t)(k & 1) : (uint32_t)((k & 1) ^ 1);
        if (!mbar_wait(&sm.empty[st], par, abort, status)) break;
        mbar_expect_tx(&sm.full[st], 4 * kTile);
        const int row = (int)(((long long)bh * a.pool_cap + sm.ids[x]) * 2) * D;
#pragma unroll
        for (int part = 0; part < 2; ++part)
#pragma unroll
          for (int hh = 0; hh < 2; ++hh)
            tma_load_2d(sm.st[st][part][hh], &tmS, &sm.full[st], 64 * hh, row + part * D);
        issued[st] = k + 1;
      }
      if (*abort) {  // let copies in flight land before the CTA exits
        for (int st = 0; st < 2; ++st)
          if (issued[st] > 0) mbar_wait(&sm.full[st], (uint32_t)((issued[st] - 1) & 1), abort, nullptr);
        mbar_wait(&sm.bar_qk, 0, abort, nullptr);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(L, D);
      bool ok = mbar_wait(&sm.bar_qk, 0, abort, status);
      if (ok) {  // P = Q K^T
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (uint32_t)(kk & 3) * 32;
          mma_bf16(tmem + COL_P, desc_kmajor_sw128(smem_u32(sm.Q[kk >> 2]) + off),
                   desc_kmajor_sw128(smem_u32(sm.st[0][0][kk >> 2]) + off), idesc, kk > 0);
        }
        mma_commit(&sm.bar_p);
        ok = mbar_wait(&sm.bar_pt, 0, abort, status);
      }
      if (ok) {  // O = Pt V: B operand V^T [j][s] sits in stage A, part 1
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (uint32_t)(kk & 3) * 32;
          mma_bf16(tmem + COL_O, desc_kmajor_sw128(smem_u32(sm.Pt[kk >> 2]) + off),
                   desc_kmajor_sw128(smem_u32(sm.st[0][1][kk >> 2]) + off), idesc, kk > 0);
        }
        mma_commit(&sm.bar_o);
        mma_commit(&sm.empty[0]);  // stage A (K, V^T) is free once these are done
      }
      for (int x = 0; ok && x < m0; ++x) {
        const int st = stage_of(x), k = x >> 1, buf = x & 1, kb = x >> 1;
        if (!mbar_wait(&sm.full[st], (uint32_t)(k & 1), abort, status)) break;
        if (!mbar_wait(&sm.acc_empty[buf], (uint32_t)((kb & 1) ^ 1), abort, status)) break;
        tc_fence_after();
        const uint32_t dcol = tmem + COL_S + 128u * buf;
        for (int part = 0; part < 2; ++part)
          for (int kk = 0; kk < 8; ++kk) {
            const uint32_t off = (uint32_t)(kk & 3) * 32;
            mma_bf16(dcol, desc_kmajor_sw128(smem_u32(sm.Q[kk >> 2]) + off),
                     desc_kmajor_sw128(smem_u32(sm.st[st][part][kk >> 2]) + off), idesc, (part | kk) > 0);
          }
        mma_commit(&sm.empty[st]);
        mma_commit(&sm.acc_full[buf]);
      }
      mma_commit(&sm.bar_done);  // every MMA issued above has completed once this fires
      mbar_wait(&sm.bar_done, 0, abort, nullptr);
    }
  } else {
    // ------------------------------------------------------------ epilogue warps
    const int ew = warp - 2;                 // 0..7
    const int quad = warp & 3;               // TMEM lane quadrant of this warp
    const int ch = (warp < 6) ? 0 : 1;       // column half
    const int t = quad * 32 + lane;          // token row of this thread
    const uint32_t lane_addr = tmem + ((uint32_t)(quad * 32) << 16);
    const int etid = ew * 32 + lane;         // 0..255
    const long long rowbase = ((long long)b * a.T + c0) * a.H + h;  // row index of token c0
    const __nv_bfloat16* vg = reinterpret_cast<const __nv_bfloat16*>(a.v);

    // the interval's boundary flags and merge indices, staged once
    if (etid < L) {
      const bool in = etid < Lc;
      sm.bnd[etid] = in ? a.boundary[(long long)bh * a.T + c0 + etid] : (uint8_t)0;
      sm.mlog[etid] = in ? a.merge_log[(long long)bh * a.T + c0 + etid] : -1;
    }
    // V^T into stage A, part 1, as the K-major B operand [j][s] (s = K index);
    // each thread issues its eight 16-byte loads before any store
    {
      constexpr int PER = L * (D / 8) / (NEPI * 32);
      uint4 raw[PER];
#pragma unroll
      for (int i = 0; i < PER; ++i) {
        const int e = etid + i * NEPI * 32;
        const int ss = e / (D / 8), j0 = (e % (D / 8)) * 8;
        raw[i] = make_uint4(0, 0, 0, 0);
        if (ss < Lc) raw[i] = *reinterpret_cast<const uint4*>(vg + (rowbase + (long long)ss * a.H) * D + j0);
      }
#pragma unroll
      for (int i = 0; i < PER; ++i) {
        const int e = etid + i * NEPI * 32;
        const int ss = e / (D / 8), j0 = (e % (D / 8)) * 8;
        const __nv_bfloat16* vv = reinterpret_cast<const __nv_bfloat16*>(&raw[i]);
        uint8_t* tile = sm.st[0][1][ss >> 6];
#pragma unroll
        for (int u = 0; u < 8; ++u)
          *reinterpret_cast<__nv_bfloat16*>(tile + sw128_offset(j0 + u, ss & 63)) = vv[u];
      }
    }
    asm volatile("bar.sync 1, 256;" ::: "memory");
    // logical slot table, one row per boundary event (one warp): row e holds
    // L(x) after the first e events of the interval; token t reads row evt[t]
    if (ew == 0) {
      int* logi = reinterpret_cast<int*>(sm.Pt[0]);  // scratch until Pt is written
      for (int x = lane; x < MAXE; x += 32) {
        logi[x] = (x < m0) ? x : -1;
        if (x < m0) sm.tab[x] = (unsigned char)x;
      }
      __syncwarp();
      unsigned long long lo64 = 0, hi64 = 0;
#pragma unroll
      for (int w4 = 0; w4 < 4; ++w4) {
        const unsigned m = __ballot_sync(0xffffffffu, sm.bnd[32 * w4 + lane] != 0);
        if (w4 < 2) lo64 |= (unsigned long long)m << (32 * w4);
        else hi64 |= (unsigned long long)m << (32 * (w4 - 2));
      }
      int nent = m0, cnt = m0, ev = 0;
      while (lo64 | hi64) {
        const int tt = lo64 ? (__ffsll((long long)lo64) - 1) : (64 + __ffsll((long long)hi64) - 1);
        if (lo64) lo64 &= lo64 - 1; else hi64 &= hi64 - 1;
        const int j = sm.mlog[tt];
        if (j >= 0) {
          for (int x = lane; x < nent; x += 32)
            if (logi[x] > j) logi[x] -= 1;
          cnt -= 1;
        }
        __syncwarp();
        if (lane == 0) logi[nent] = cnt;
        nent += 1;
        cnt += 1;
        ev += 1;
        __syncwarp();
        for (int x = lane; x < nent; x += 32) sm.tab[ev * MAXE + x] = (unsigned char)logi[x];
        __syncwarp();
      }
    }
    // events at or before each token, and the entry holding it
    if (etid < L) {  // warps 2..5, one token per lane
      const int tt = etid;
      int e = 0;
#pragma unroll
      for (int w4 = 0; w4 < 4; ++w4) {
        const unsigned m = __ballot_sync(0xffffffffu, sm.bnd[32 * w4 + lane] != 0);
        if (32 * w4 + 31 <= tt) e += __popc(m);
        else if (32 * w4 <= tt) e += __popc(m & (0xffffffffu >> (31 - (tt - 32 * w4))));
      }
      sm.evt[tt] = e;
      sm.ent[tt] = (e == 0) ? m0 - 1 : m0 + e - 1;
    }
    asm volatile("bar.sync 1, 256;" ::: "memory");
    const float* lam_t = (a.lam && t < Lc) ? a.lam + (rowbase + (long long)t * a.H) * C : nullptr;
    const int evt_t = sm.evt[t];
    // ---- Pt = P * lambda_{t, L_t(e(s))} for s <= t (bf16), s in this warp's half
    if (mbar_wait(&sm.bar_p, 0, abort, status)) {
      tc_fence_after();
      float p[64];
      tmem_ld32(lane_addr + COL_P + 64 * ch, p);
      tmem_ld32(lane_addr + COL_P + 64 * ch + 32, p + 32);
      uint8_t* tile = sm.Pt[ch];
#pragma unroll
      for (int c8 = 0; c8 < 8; ++c8) {
        uint32_t packed[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          float w2[2];
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const int sl = c8 * 8 + 2 * i + u;  // column inside the half
            const int ss = 64 * ch + sl;
            float w = 0.f;
            if (ss <= t && t < Lc) {
              const int li = sm.tab[evt_t * MAXE + sm.ent[ss]];
              w = lam_t ? lam_t[li] : 1.f;
            }
            w2[u] = p[sl] * w;
          }
          __nv_bfloat162 pr = __floats2bfloat162_rn(w2[0], w2[1]);
          packed[i] = *reinterpret_cast<uint32_t*>(&pr);
        }
        *reinterpret_cast<uint4*>(tile + t * 128 + (((c8 ^ (t & 7)) & 7) << 4)) =
            make_uint4(packed[0], packed[1], packed[2], packed[3]);
      }
    }
    fence_proxy_async();
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(&sm.bar_pt);
    // ---- o = O_intra + sum_x lambda_{t, L_t(x)} D_x
    float o[64];
#pragma unroll
    for (int i = 0; i < 64; ++i) o[i] = 0.f;
    if (mbar_wait(&sm.bar_o, 0, abort, status)) {
      tc_fence_after();
      tmem_ld32(lane_addr + COL_O + 64 * ch, o);
      tmem_ld32(lane_addr + COL_O + 64 * ch + 32, o + 32);
    }
    // weight of state x for this token; fetched one state ahead of its use
    auto weight = [&](int x) -> float {
      if (t >= Lc || x >= m0) return 0.f;
      return lam_t ? lam_t[sm.tab[evt_t * MAXE + x]] : 1.f;
    };
    float w_next = weight(0);
    for (int x = 0; x < m0; ++x) {
      const int buf = x & 1, kb = x >> 1;
      const float w = w_next;
      w_next = weight(x + 1);
      if (!mbar_wait(&sm.acc_full[buf], (uint32_t)(kb & 1), abort, status)) break;
      tc_fence_after();
      float dv[32];
      const uint32_t base = lane_addr + COL_S + 128u * buf + 64 * ch;
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
  CUtensorMap mq, mk, ms;
  const long long rows = (long long)a.B * a.H * a.pool_cap * 2 * D;
  if (!map_tokens(&mq, a.q, a.B, a.T, a.H) || !map_tokens(&mk, a.k, a.B, a.T, a.H) || !map_pool(&ms, a.pool, rows))
    return cudaErrorInvalidValue;
  const size_t smem = sizeof(TcSmem) + 1024;
  cudaError_t e = cudaFuncSetAttribute(readout_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(a.nsnap, a.B * a.H);
  readout_tc_kernel<<<grid, NT, smem, st>>>(a, mq, mk, ms, status);
  return cudaGetLastError();
}

size_t readout_tc_smem_bytes() { return sizeof(TcSmem) + 1024; }

}  // namespace dla
