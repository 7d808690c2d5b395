// Backward pass of thin-key attention (the training path): dQ and dK are r
// wide, dV is d_v wide.
//
// Paper: Section 2.1, Eqs. 1-4 (the forward being differentiated); training
// with thin keys is Sections 3.2-3.3.  Per head, with s = scale q k^T (masked),
// p = softmax(s), out = p v and dL/d(out) = dO:
//     dV = p^T dO,   dP = dO v^T,   dS = p * (dP - D),  D_i = sum_c dO_ic out_ic,
//     dQ = scale dS k,   dK = scale dS^T q
// (D_i equals rowsum(dP * p) for the exact forward output).
//
// Two kernels:
//   bwd_prep: -D = -rowsum(dO * out) and -lse log2(e) per query row (rows
//     padded to a multiple of 128), and dQ set to zero.
//   the gradient kernel: for r <= 64 the tensor-memory kernel of
//     backward_tc.cu; for r = 128 (whose TMEM accumulators do not fit beside
//     the score tiles) bwd_main below.
//   bwd_main: one CTA per (sequence, kv head g, 64-key tile j); 4 warps, warp
//     w owns keys 16w..16w+15 of the tile.  It visits every query tile i (64
//     rows; i >= j when causal) of each of the G query heads of g and, on the
//     tensor cores with mma.sync.m16n8k16 (bf16 operands, fp32 accumulation):
//         S^T = K Q^T and P^T = exp2(S^T scale log2e - lse log2e)   (recomputed)
//         dP^T = V dO^T,  dS^T = P^T * (dP^T - D)
//         dV += P^T dO,   dK += dS^T Q                     (registers, whole run)
//         dQ(i) += dS K   (per-warp partials in shared memory, summed and added
//                          to global dQ with float4 atomics, once per query part)
//     P^T and dS^T go from the accumulator layout straight into the A operand
//     of the next products; dS is transposed for dQ with movmatrix.  Q, dO and
//     the per-row statistics stream through a double-buffered cp.async ring
//     with XOR-swizzled rows (conflict-free ldmatrix); rows past S are zero
//     filled.
#include <cuda_bf16.h>

#include "common.cuh"
#include "kernels.h"

namespace tk {
namespace {

constexpr int kTile = 64;       // keys per CTA, queries per visit
constexpr int kBwdThreads = 128;

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& a, uint32_t& b, uint32_t& c,
                                        uint32_t& d) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a), "=r"(b), "=r"(c), "=r"(d)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& a, uint32_t& b, uint32_t& c,
                                          uint32_t& d) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a), "=r"(b), "=r"(c), "=r"(d)
               : "r"(addr));
}
__device__ __forceinline__ uint32_t movm_t(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}
// d (16x8 fp32) += A (16x16 bf16, row) * B (16x8 bf16, col)
__device__ __forceinline__ void mma16816(float* d, uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Byte offset of 16-byte chunk c of row `row` in a tile whose rows are W bytes:
// the chunk index is XORed with a few row bits so that the 8 rows one
// ldmatrix 8x8 read touches fall in 8 different 16-byte bank groups.
template <int W>
__device__ __forceinline__ uint32_t swz(int row, int c) {
  constexpr int C = W / 16;
  int pc;
  if constexpr (C >= 8) pc = c ^ (row & 7);
  else if constexpr (C == 4) pc = c ^ ((row >> 1) & 3);
  else pc = c ^ ((row >> 2) & 1);
  return static_cast<uint32_t>(row * W + pc * 16);
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
               "r"(valid ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src, bool valid) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src),
               "r"(valid ? 4 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Copy `rows` valid rows of W bytes (a 64-row tile, row stride W in global
// memory) into the swizzled tile at `dst`; rows past `rows` are zero filled.
template <int W>
__device__ __forceinline__ void load_tile(uint32_t dst, const unsigned char* src, int rows, int tid) {
  constexpr int C = W / 16;
  for (int e = tid; e < kTile * C; e += kBwdThreads) {
    const int row = e / C, c = e % C;
    const bool valid = row < rows;
    cp_async16(dst + swz<W>(row, c), src + (valid ? static_cast<size_t>(row) * W + c * 16 : 0), valid);
  }
}

// ---------------------------------------------------------------- preprocessing
// DV / 8 threads per padded statistics row (b, h, i < S_pad), 16 bytes of out
// and of d_out each: for i < S, nd = -sum_c dO * out (fp32), nl2 = -lse *
// log2(e) and the row of dQ zeroed; for S <= i < S_pad, nd = 0 and nl2 = -inf
// (such rows get softmax weight 0).
constexpr int kPrepThreads = 256;
template <int R, int DV>
__global__ void __launch_bounds__(kPrepThreads) bwd_prep(const BackwardParams p) {
  constexpr int TPR = DV / 8;                       // threads per row
  constexpr int RPB = kPrepThreads / TPR;           // rows per block
  static_assert(32 % TPR == 0, "a row's threads sit in one warp");
  const int sub = threadIdx.x % TPR;
  const long long row = static_cast<long long>(blockIdx.x) * RPB + threadIdx.x / TPR;
  const long long rows = static_cast<long long>(p.B) * p.Hq * p.S_pad;
  // no lane leaves before the shuffle below: a warp holds several rows
  const bool in_grid = row < rows;
  const long long bh = in_grid ? row / p.S_pad : 0;
  const int i = in_grid ? static_cast<int>(row - bh * p.S_pad) : 0;
  const bool real = in_grid && i < p.S;
  const long long x = bh * p.S + i;   // row of the [B][Hq][S] tensors
  float acc = 0.f;
  if (real) {
    const uint4 o = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p.out) + x * DV)[sub];
    const uint4 d = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p.d_out) + x * DV)[sub];
    const uint32_t ow[4] = {o.x, o.y, o.z, o.w}, dw[4] = {d.x, d.y, d.z, d.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) acc += bf16lo(ow[e]) * bf16lo(dw[e]) + bf16hi(ow[e]) * bf16hi(dw[e]);
  }
#pragma unroll
  for (int off = TPR / 2; off >= 1; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
  if (!in_grid) return;
  if (sub == 0) {
    p.nd[row] = real ? -acc : 0.f;
    p.nl2[row] = real ? -p.lse[x] * 1.4426950408889634f : -INFINITY;
  }
  if (!real) return;
  float4* dq = reinterpret_cast<float4*>(p.dq + x * R);
#pragma unroll
  for (int c = sub; c < R / 4; c += TPR) dq[c] = make_float4(0.f, 0.f, 0.f, 0.f);
}

// ---------------------------------------------------------------- main kernel
template <int R, int DV>
struct BCfg {
  static constexpr int KW = R * 2, VW = DV * 2;   // bytes per K / Q row and V / dO row
  // queries per step of a visit: the S^T / dP^T fragments of a step are held at once
  // (32 fits in registers up to r = 64; at r = 128 the dK / dQ fragments leave room for 16)
  static constexpr int PQ = R <= 64 ? 32 : 16, PARTS = kTile / PQ;
  static constexpr int OFF_K = 0;
  static constexpr int OFF_V = OFF_K + kTile * KW;
  static constexpr int OFF_BUF = OFF_V + kTile * VW;
  static constexpr int BUF_Q = 0, BUF_DO = kTile * KW, BUF_LSE = BUF_DO + kTile * VW,
                       BUF_D = BUF_LSE + kTile * 4, BUF = BUF_D + kTile * 4;
  // dQ partials of one part of the queries, one buffer per warp, rows padded to R + 8
  // floats so that a warp's 64-bit fragment stores hit 32 different banks
  static constexpr int DQP = R + 8;
  static constexpr int OFF_DQ = OFF_BUF + 2 * BUF;          // [4 warps][PQ][DQP] fp32
  static constexpr int SMEM = OFF_DQ + 4 * PQ * DQP * 4;
  static_assert(SMEM <= 227 * 1024, "shared memory");
};

template <int R, int DV>
__global__ void __launch_bounds__(kBwdThreads, 1) bwd_main(const BackwardParams p) {
  using C = BCfg<R, DV>;
  extern __shared__ __align__(128) unsigned char smem[];
  const uint32_t sbase = smem_addr(smem);
  float* dqw = reinterpret_cast<float*>(smem + C::OFF_DQ);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g8 = lane >> 2, t4 = lane & 3;          // fragment row / column pair
  const int mi = lane >> 3, rr = lane & 7;          // ldmatrix: matrix, row within it
  const int S = p.S, G = p.Hq / p.Hkv;
  const int n_t = (S + kTile - 1) / kTile;
  const int j = static_cast<int>(blockIdx.x % n_t);
  const int bg = static_cast<int>(blockIdx.x / n_t);
  const int b = bg / p.Hkv, g = bg % p.Hkv;
  const int i0 = p.causal ? j : 0;
  const int per_head = n_t - i0;
  const int visits = G * per_head;
  const float sl2 = p.scale * 1.4426950408889634f;

  // this CTA's keys and values, once
  {
    const size_t kv = static_cast<size_t>(b) * p.Hkv + g;
    const int rows = min(kTile, S - j * kTile);
    load_tile<C::KW>(sbase + C::OFF_K,
                     static_cast<const unsigned char*>(p.k) + (kv * S + j * kTile) * C::KW, rows, tid);
    load_tile<C::VW>(sbase + C::OFF_V,
                     static_cast<const unsigned char*>(p.v) + (kv * S + j * kTile) * C::VW, rows, tid);
  }
  auto load_visit = [&](int vis, int buf) {
    const int h = g * G + vis / per_head, i = i0 + vis % per_head;
    const size_t qrow = (static_cast<size_t>(b) * p.Hq + h) * S + static_cast<size_t>(i) * kTile;
    const int rows = min(kTile, S - i * kTile);
    const uint32_t bb = sbase + C::OFF_BUF + buf * C::BUF;
    load_tile<C::KW>(bb + C::BUF_Q, static_cast<const unsigned char*>(p.q) + qrow * C::KW, rows, tid);
    load_tile<C::VW>(bb + C::BUF_DO, static_cast<const unsigned char*>(p.d_out) + qrow * C::VW, rows, tid);
    {  // the rows' statistics (padded rows: always in range): threads 0-63 nl2, 64-127 nd
      const int r = tid & (kTile - 1);
      const size_t srow = (static_cast<size_t>(b) * p.Hq + h) * p.S_pad + static_cast<size_t>(i) * kTile + r;
      cp_async4(bb + (tid < kTile ? C::BUF_LSE : C::BUF_D) + r * 4, (tid < kTile ? p.nl2 : p.nd) + srow, true);
    }
  };
  if (visits > 0) load_visit(0, 0);
  cp_async_commit();

  float dv_acc[DV / 8][4], dk_acc[R / 8][4];
#pragma unroll
  for (int n = 0; n < DV / 8; ++n) dv_acc[n][0] = dv_acc[n][1] = dv_acc[n][2] = dv_acc[n][3] = 0.f;
#pragma unroll
  for (int n = 0; n < R / 8; ++n) dk_acc[n][0] = dk_acc[n][1] = dk_acc[n][2] = dk_acc[n][3] = 0.f;
  const int krow = warp * 16;                       // this warp's first key in the tile
  const int key0 = j * kTile + krow + g8;           // absolute keys of fragment rows g8, g8 + 8

  for (int vis = 0; vis < visits; ++vis) {
    const int cur = vis & 1;
    if (vis + 1 < visits) load_visit(vis + 1, cur ^ 1);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    const int h = g * G + vis / per_head, i = i0 + vis % per_head;
    const uint32_t bq = sbase + C::OFF_BUF + cur * C::BUF + C::BUF_Q;
    const uint32_t bdo = sbase + C::OFF_BUF + cur * C::BUF + C::BUF_DO;
    const float* nl2 = reinterpret_cast<const float*>(smem + C::OFF_BUF + cur * C::BUF + C::BUF_LSE);
    const float* nd = reinterpret_cast<const float*>(smem + C::OFF_BUF + cur * C::BUF + C::BUF_D);
    const bool diag = p.causal && i == j;

#pragma unroll 1
    for (int part = 0; part < C::PARTS; ++part) {
      const int qb = part * C::PQ;                 // first query (in the tile) of this part
      float sa[C::PQ / 8][4], dp[C::PQ / 8][4];
#pragma unroll
      for (int n = 0; n < C::PQ / 8; ++n) sa[n][0] = sa[n][1] = sa[n][2] = sa[n][3] = dp[n][0] = dp[n][1] = dp[n][2] = dp[n][3] = 0.f;
      // ---- S^T = K Q^T (16 keys x PQ queries), k = r
#pragma unroll
      for (int ks = 0; ks < R / 16; ++ks) {
        uint32_t a0, a1, a2, a3;
        ldsm_x4(sbase + C::OFF_K + swz<C::KW>(krow + (mi & 1) * 8 + rr, 2 * ks + (mi >> 1)), a0, a1, a2, a3);
#pragma unroll
        for (int np = 0; np < C::PQ / 16; ++np) {
          uint32_t b0, b1, b2, b3;  // queries qb+16np.. : (n-tile 2np, k lo/hi), (2np+1, k lo/hi)
          ldsm_x4(bq + swz<C::KW>(qb + 16 * np + (mi >> 1) * 8 + rr, 2 * ks + (mi & 1)), b0, b1, b2, b3);
          mma16816(sa[2 * np], a0, a1, a2, a3, b0, b1);
          mma16816(sa[2 * np + 1], a0, a1, a2, a3, b2, b3);
        }
      }
      // ---- dP^T = V dO^T (16 keys x PQ queries), k = d_v
#pragma unroll
      for (int ks = 0; ks < DV / 16; ++ks) {
        uint32_t a0, a1, a2, a3;
        ldsm_x4(sbase + C::OFF_V + swz<C::VW>(krow + (mi & 1) * 8 + rr, 2 * ks + (mi >> 1)), a0, a1, a2, a3);
#pragma unroll
        for (int np = 0; np < C::PQ / 16; ++np) {
          uint32_t b0, b1, b2, b3;
          ldsm_x4(bdo + swz<C::VW>(qb + 16 * np + (mi >> 1) * 8 + rr, 2 * ks + (mi & 1)), b0, b1, b2, b3);
          mma16816(dp[2 * np], a0, a1, a2, a3, b0, b1);
          mma16816(dp[2 * np + 1], a0, a1, a2, a3, b2, b3);
        }
      }
      // ---- P^T and dS^T in the accumulator layout: (key g8 | g8+8, query 2t4 | 2t4+1)
#pragma unroll
      for (int n = 0; n < C::PQ / 8; ++n) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int q = qb + 8 * n + 2 * t4 + (e & 1);     // query in the tile
          const int key = key0 + (e >> 1) * 8;              // absolute key
          const bool hide = diag && key > i * kTile + q;
          const float pr = hide ? 0.f : fast_exp2(fmaf(sa[n][e], sl2, nl2[q]));
          sa[n][e] = pr;
          dp[n][e] = pr * (dp[n][e] + nd[q]);
        }
      }
      // A operands (16 keys x 16 queries) of P^T and dS^T for each 16-query k-step
      uint32_t pa[C::PQ / 16][4], da[C::PQ / 16][4];
#pragma unroll
      for (int kk = 0; kk < C::PQ / 16; ++kk) {
        pa[kk][0] = pack_bf16(sa[2 * kk][0], sa[2 * kk][1]);
        pa[kk][1] = pack_bf16(sa[2 * kk][2], sa[2 * kk][3]);
        pa[kk][2] = pack_bf16(sa[2 * kk + 1][0], sa[2 * kk + 1][1]);
        pa[kk][3] = pack_bf16(sa[2 * kk + 1][2], sa[2 * kk + 1][3]);
        da[kk][0] = pack_bf16(dp[2 * kk][0], dp[2 * kk][1]);
        da[kk][1] = pack_bf16(dp[2 * kk][2], dp[2 * kk][3]);
        da[kk][2] = pack_bf16(dp[2 * kk + 1][0], dp[2 * kk + 1][1]);
        da[kk][3] = pack_bf16(dp[2 * kk + 1][2], dp[2 * kk + 1][3]);
      }
      // ---- dV += P^T dO (16 keys x d_v), k = PQ queries
#pragma unroll
      for (int kk = 0; kk < C::PQ / 16; ++kk) {
#pragma unroll
        for (int np = 0; np < DV / 16; ++np) {
          uint32_t b0, b1, b2, b3;  // (d_v n-tile 2np: queries lo, hi), (2np+1: lo, hi)
          ldsm_x4_t(bdo + swz<C::VW>(qb + 16 * kk + (mi & 1) * 8 + rr, 2 * np + (mi >> 1)), b0, b1, b2, b3);
          mma16816(dv_acc[2 * np], pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3], b0, b1);
          mma16816(dv_acc[2 * np + 1], pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3], b2, b3);
        }
      }
      // ---- dK += dS^T Q (16 keys x r), k = PQ queries (scale applied at the end)
#pragma unroll
      for (int kk = 0; kk < C::PQ / 16; ++kk) {
#pragma unroll
        for (int np = 0; np < R / 16; ++np) {
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(bq + swz<C::KW>(qb + 16 * kk + (mi & 1) * 8 + rr, 2 * np + (mi >> 1)), b0, b1, b2, b3);
          mma16816(dk_acc[2 * np], da[kk][0], da[kk][1], da[kk][2], da[kk][3], b0, b1);
          mma16816(dk_acc[2 * np + 1], da[kk][0], da[kk][1], da[kk][2], da[kk][3], b2, b3);
        }
      }
      // ---- dQ += dS K (PQ queries x r), k = this warp's 16 keys: dS via movmatrix;
      // the warp's partial goes to its own buffer, the four are summed below
      float* mine = dqw + warp * C::PQ * C::DQP;
#pragma unroll
      for (int mt = 0; mt < C::PQ / 16; ++mt) {
        const uint32_t a0 = movm_t(da[mt][0]);   // queries 16mt+g8,   keys 2t4..   (key block 0-7)
        const uint32_t a1 = movm_t(da[mt][2]);   // queries 16mt+8+g8, keys 2t4..
        const uint32_t a2 = movm_t(da[mt][1]);   // queries 16mt+g8,   keys 8+2t4..
        const uint32_t a3 = movm_t(da[mt][3]);   // queries 16mt+8+g8, keys 8+2t4..
#pragma unroll
        for (int np = 0; np < R / 16; ++np) {
          uint32_t b0, b1, b2, b3;  // B[key][r] = K: (r n-tile 2np: keys lo, hi), (2np+1: lo, hi)
          ldsm_x4_t(sbase + C::OFF_K + swz<C::KW>(krow + (mi & 1) * 8 + rr, 2 * np + (mi >> 1)), b0, b1, b2, b3);
          float c0[4] = {0.f, 0.f, 0.f, 0.f}, c1[4] = {0.f, 0.f, 0.f, 0.f};
          mma16816(c0, a0, a1, a2, a3, b0, b1);
          mma16816(c1, a0, a1, a2, a3, b2, b3);
          const int q0 = 16 * mt + g8;            // query within the half
          const int r0 = 16 * np + 2 * t4;
          *reinterpret_cast<float2*>(mine + q0 * C::DQP + r0) = make_float2(c0[0], c0[1]);
          *reinterpret_cast<float2*>(mine + (q0 + 8) * C::DQP + r0) = make_float2(c0[2], c0[3]);
          *reinterpret_cast<float2*>(mine + q0 * C::DQP + r0 + 8) = make_float2(c1[0], c1[1]);
          *reinterpret_cast<float2*>(mine + (q0 + 8) * C::DQP + r0 + 8) = make_float2(c1[2], c1[3]);
        }
      }
      __syncthreads();
      // the part's dQ: the four warps' partials summed, added into dq (4 floats at a time)
      {
        const int rows = min(C::PQ, S - i * kTile - qb);
        float* dq = p.dq + ((static_cast<size_t>(b) * p.Hq + h) * S + static_cast<size_t>(i) * kTile + qb) * R;
#pragma unroll 1
        for (int e = tid * 4; e < C::PQ * R; e += kBwdThreads * 4) {
          const int q = e / R, c = e % R;
          if (q >= rows) continue;
          float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
          for (int w = 0; w < 4; ++w) {
            const float4 x = *reinterpret_cast<const float4*>(dqw + (w * C::PQ + q) * C::DQP + c);
            sum.x += x.x; sum.y += x.y; sum.z += x.z; sum.w += x.w;
          }
          sum.x *= p.scale; sum.y *= p.scale; sum.z *= p.scale; sum.w *= p.scale;
          atomicAdd(reinterpret_cast<float4*>(dq + e), sum);
        }
      }
      __syncthreads();
    }
  }
  cp_async_wait<0>();

  // dK (times the softmax scale) and dV of this warp's 16 keys
  const size_t kv = static_cast<size_t>(b) * p.Hkv + g;
#pragma unroll
  for (int hh = 0; hh < 2; ++hh) {
    const int key = key0 + hh * 8;
    if (key >= S) continue;
    float* dk = p.dk + (kv * S + key) * R;
    float* dv = p.dv + (kv * S + key) * DV;
#pragma unroll
    for (int n = 0; n < R / 8; ++n)
      *reinterpret_cast<float2*>(dk + 8 * n + 2 * t4) =
          make_float2(dk_acc[n][2 * hh] * p.scale, dk_acc[n][2 * hh + 1] * p.scale);
#pragma unroll
    for (int n = 0; n < DV / 8; ++n)
      *reinterpret_cast<float2*>(dv + 8 * n + 2 * t4) = make_float2(dv_acc[n][2 * hh], dv_acc[n][2 * hh + 1]);
  }
}

template <int R, int DV>
cudaError_t launch_t(const BackwardParams& p, cudaStream_t s, int* uns) {
  const long long rows = static_cast<long long>(p.B) * p.Hq * p.S_pad;
  constexpr int rpb = kPrepThreads / (DV / 8);
  const long long pblocks = (rows + rpb - 1) / rpb;
  if (pblocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  bwd_prep<R, DV><<<static_cast<unsigned>(pblocks), kPrepThreads, 0, s>>>(p);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if constexpr (R <= 64) {
    return launch_backward_tc(p, s, uns);
  } else {
    using C = BCfg<R, DV>;
    e = cudaFuncSetAttribute(bwd_main<R, DV>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    const long long n_t = (p.S + kTile - 1) / kTile;
    const long long grid = static_cast<long long>(p.B) * p.Hkv * n_t;
    if (grid > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    bwd_main<R, DV><<<static_cast<unsigned>(grid), kBwdThreads, C::SMEM, s>>>(p);
    return cudaGetLastError();
  }
}

template <int R>
cudaError_t by_dv(const BackwardParams& p, cudaStream_t s, int* uns) {
  switch (p.DV) {
    case 64: return launch_t<R, 64>(p, s, uns);
    case 128: return launch_t<R, 128>(p, s, uns);
  }
  *uns = 1;
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_backward(const BackwardParams& p, cudaStream_t stream, int* unsupported) {
  *unsupported = 0;
  switch (p.R) {
    case 16: return by_dv<16>(p, stream, unsupported);
    case 32: return by_dv<32>(p, stream, unsupported);
    case 64: return by_dv<64>(p, stream, unsupported);
    case 128: return by_dv<128>(p, stream, unsupported);
  }
  *unsupported = 1;
  return cudaSuccess;
}

}  // namespace tk
