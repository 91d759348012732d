// A whole round of local steps of a two-layer bf16 MLP (input -> H hidden
// ReLU units -> 10 classes) in ONE launch (Eq. 4, "otherwise" branch: each
// worker runs tau_i SGD steps from the global model).
//
// One thread-block cluster serves one worker at a time.  The hidden units come in
// groups of 128 (one tensor-core tile of rows); each group is served by S
// CTAs (S = 1 or 2) that split the INPUT dimension: CTA h of the group owns
// input columns [c_h, c_{h+1}) of the group's 128 rows of W0 (a split on a
// 64-column K-block boundary).  Cluster rank = group * S + h.
//
// The worker's model stays on chip for the whole round.  A CTA keeps its
// block of W0 twice: the fp32 master values in tensor memory (TMEM lane =
// hidden unit, column = input column) and their bf16 copy, the A operand of
// the forward GEMM, in shared memory (K-major, 128-byte swizzled K-blocks).
// Its head-weight columns, its b0 entries and a private copy of the head
// bias (updated identically by every CTA) live in shared memory.  The model
// is read from the global slot once, before the first step (the W0 block by
// TMA: fp32 tiles staged in shared memory on their way to TMEM; the bf16
// operand is then rounded from TMEM), and the worker's replica is written
// once, in the last step (the weight-gradient epilogue stages the updated W0
// columns in shared memory and TMA stores them).  Per step only the
// mini-batch (staged bf16 X and X^T tiles, by TMA) and the labels come from
// global memory.
//
// Every step of the worker runs inside the cluster:
//
//  F  forward: each CTA computes the partial pre-activation of the group's
//     128 units over its own input columns on tcgen05 (resident W0; the
//     first X tiles are prefetched during the previous step).  With S = 2
//     each CTA keeps 128/S of the units: the epilogue stores its own units'
//     partials locally and writes the partner's straight into the partner's
//     incoming buffer with asynchronous 16-byte stores (st.async, distributed
//     shared memory) that complete on the partner's mbarrier (a pairwise
//     wait instead of a cluster barrier); then
//     z = (part_0 + part_1) + b0, h = relu(z), bf16;
//  H  last layer for the CTA's units: partial logits (double-buffered by
//     step parity), summed over the whole cluster in rank order through
//     distributed shared memory after one cluster barrier, softmax
//     cross-entropy; the masked input gradient dz0[b][u] of its units is
//     written (as bf16, 16-byte chunks of 8 samples) into the
//     128-byte-swizzled K-major dz0^T tile (the A operand of step D); bias
//     gradient and SGD of b0 (own units), of the head weights (own columns)
//     and of the head bias.  With S = 2, once the CTA has read h for the
//     last time in the step, its dz0^T rows go to the partner with st.async,
//     completing on the partner's mbarrier, which the partner's MMA issuers
//     wait on before step D (a pairwise wait, no cluster barrier);
//  D  weight gradient of the group's 128 rows over the CTA's own input
//     columns, dW0[o][k] = sum_b dz0[b][o] X[b][k], on tcgen05 in 48-column
//     tiles (the last one 16 or 32 columns; X^T tiles of 48 rows by TMA into
//     a four-deep ring, two slots per issuing chain, the first ones during
//     step F).  The tiles alternate between two chains, each with its own
//     issuing thread, TMEM buffer and epilogue warpgroup, so that one chain's
//     MMA issue overlaps the other's epilogue; the epilogue reads the
//     gradient and the fp32 master from TMEM, applies W0 <- W0 - lr dW0,
//     stores the master back to TMEM and its bf16 copy into the resident A
//     operand (in the worker's last step: into the replica slot instead).
//
// Ownership: a CTA rewrites only its own block of W0, its own b0 entries and
// head-weight columns, and its private head bias, so its next step reads its
// own writes.  The logits it reads from other CTAs follow the cluster
// barrier of the step; each buffer of partial logits is rewritten two steps
// later, after the next step's barrier, which every reader has passed.  The
// partner's partials and dz0 rows arrive on mbarriers (expected bytes set at
// the start of each step).  The incoming partials land in the h tile: the
// partner writes them in its next forward epilogue, which follows its step
// D, which waits for this CTA's dz0 rows, which this CTA sends only after its
// last read of h; so they never overwrite h in use.  A final cluster barrier
// keeps every CTA resident until no peer can read its partial logits.
// Generic-proxy writes that the tensor core reads are fenced with
// fence.proxy.async.  Arithmetic and rounding points are those of the
// per-layer path (the pair's two partial sums are added in rank order).
//
// The staging of the next round into the other input buffer runs beside
// the kernel at a lower launch priority, on the SMs its clusters leave free.
//
// The grid has one cluster per worker, or as many clusters as fit on the GPU
// at once when there are more workers; a table gives each cluster its
// workers, which it runs one after the other (the host deals them by
// decreasing tau to the cluster with the least work so far).
//
// Warp roles (384 threads): warp 0 lane 0 issues TMA, warp 1 lane 0 issues
// tcgen05.mma (in step D warps 1 and 3 issue one chain each), warp 2 owns the
// TMEM allocation (all 512 columns: one CTA per SM), warps 4..11 are the two
// epilogue warpgroups (each covering the 128 TMEM lanes), all warps share the
// CUDA-core work of step H.
//
// TMEM columns: [0, kTAcc) fp32 master of the W0 block (416 columns); [kTAcc,
// 512) the forward accumulator (B columns), the last layer's accumulators
// and, in step D, the two 48-column weight-gradient buffers (the uses never
// overlap in time).
#include "common.cuh"
#include "internal.h"

namespace oscars {
namespace {

constexpr int kFT = 384;               // threads
constexpr int kFU = 128;               // hidden units per group (tensor-core rows)
constexpr int kFC = 10;                // classes
constexpr int kFMaxCluster = 8;
constexpr int kFBK = 64;               // K-block (bf16 elements, 128 bytes)
constexpr int kND = 32;                // columns per fp32 model tile (the load)
// replica staging of the last step, per epilogue warp: two 32 x 32 fp32
// boxes and two 32 x 16 boxes (1024-byte aligned for the swizzled ones)
constexpr int kStg32 = 32 * 32 * 4, kStg16 = 32 * 16 * 4;
constexpr int kStgBytes = 2 * kStg32 + 2 * kStg16;
constexpr int kDT = 48;                // columns per weight-gradient tile
constexpr int kNBD = 2;                // weight-gradient TMEM buffers (one per issuing chain)
constexpr int kNXD = 4;                // X^T tile buffers in shared memory (even: two per issuing chain)
constexpr int kTAcc = 512 - kNBD * kDT;   // first TMEM column of the accumulators = master columns (416)
constexpr int kMaxKb = (kTAcc + kFBK - 1) / kFBK;   // resident K-blocks of W0
constexpr int kW0Blk = kFU * kFBK * 2; // one resident K-block: 128 rows x 64 columns bf16
static_assert((kFT / 32 - 4) * kStgBytes <= kMaxKb * kW0Blk && kStgBytes % 1024 == 0 && kStg32 % 1024 == 0,
              "the replica staging of the epilogue warps fits the resident-operand area, 1024-byte aligned");

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long v;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(v));
  return v;
}

// byte offset of element (row, k) in a K-major 128-byte-swizzled tile of one
// 64-wide K-block (the layout TMA writes and UMMA reads)
__device__ __forceinline__ uint32_t sw128_offset(int row, int k) {
  return static_cast<uint32_t>((row >> 3) * 1024 + (row & 7) * 128 + ((((k >> 3) ^ (row & 7)) & 7) << 4) +
                               (k & 7) * 2);
}

// one bf16 value (round to nearest even) at a byte address of shared memory
__device__ __forceinline__ void st_bf16(uint8_t* p, float v) {
  *reinterpret_cast<__nv_bfloat16*>(p) = __float2bfloat16_rn(v);
}

// bf16 copy of columns [c0, c0 + N) of row r (c0 a multiple of 8) into the
// resident W0 operand: one 16-byte chunk of a swizzled 128-byte row per 8
// columns, each in the K-block of its columns
template <int N>
__device__ __forceinline__ void put_w0_cols(uint8_t* w0s, int r, int c0, const float (&v)[N]) {
#pragma unroll
  for (int i = 0; i < N / 8; ++i) {
    const int col = c0 + 8 * i;
    *reinterpret_cast<uint4*>(w0s + (col / kFBK) * kW0Blk + sw128_offset(r, col % kFBK)) =
        make_uint4(pack_bf16x2(v[8 * i], v[8 * i + 1]), pack_bf16x2(v[8 * i + 2], v[8 * i + 3]),
                   pack_bf16x2(v[8 * i + 4], v[8 * i + 5]), pack_bf16x2(v[8 * i + 6], v[8 * i + 7]));
  }
}

// Per-shape configuration (all sizes known at compile time).
template <int B, int S>
struct FCfg {
  static_assert(B == 32 || B == 64, "batch of 32 or 64");
  static_assert(S == 1 || S == 2, "one or two CTAs per group");
  static_assert(kTAcc + B <= 512, "the forward accumulator must fit the accumulator columns");
  static constexpr int kUPC = kFU / S;                      // units per CTA in steps F (kept) and H
  // the last layer's three products on the tensor core (batch 64, two CTAs
  // per group; see the operand tiles below)
  static constexpr bool kTCH = B == 64 && S == 2;
  static constexpr int kStagesF = kTCH ? 5 : 4;
  static constexpr int kBBytes = B * kFBK * 2;              // X tile: B rows x 64 k
  static constexpr int kXtBytes = kDT * kFBK * 2;           // X^T tile: 48 rows x 64 k (K padded)
  static constexpr int kDRing = kNXD * kXtBytes;
  static constexpr int kFRing = kStagesF * kBBytes;
  static constexpr int kZs = B + 4;                         // row stride of the partial z exchange (floats)
  static constexpr int kZBytes = S > 1 ? kUPC * kZs * 4 : 0;  // own partials (the incoming ones alias hs)
  static constexpr int kZTx = kUPC * B * 4;                 // partial bytes the partner sends per step
  static constexpr int kDzTx = kUPC * B * 2;                // dz0^T bytes the partner sends per step
  static constexpr int kRegion = kDRing + (kFRing > kZBytes ? kFRing : kZBytes);   // D ring | F ring or z
  static constexpr int kDzT = kFU * 128;                    // dz0^T tile: 128 rows x 64 k (batch padded)
  static constexpr int kTpr = 256 / B;                      // threads per row, partial logits
  static constexpr int kHsd = kUPC + 4 * kTpr;              // padded row stride of the float h tile
  static constexpr int kChunks = B / 8;                     // 8-sample chunks of a dz0^T row
  static constexpr int kW1Items = kFC * (kUPC / 4);         // (class, 4 units) items of the head update
  // the last layer's three products on the tensor core (batch 64, two CTAs
  // per group): operand tiles of 128-byte K-major rows in the forward X ring,
  // which is idle between the forward's partial sums and step D.  An A tile
  // holds 64 used rows; the MMA (M = 128) also reads the next 64 rows, which
  // feed accumulator lanes nobody reads and may lie past the ring, in the
  // resident W0 area that follows it.  dz1 takes h's slot once the logits
  // MMA has completed.
  static constexpr int tH = 0;                               // h [b][u]: logits A (rows b)
  static constexpr int tHT = 8192;                           // h^T [u][b]: head-gradient A (rows u)
  static constexpr int tDzT = 16384;                         // dz1^T [c][b]: head-gradient B (16 rows)
  static constexpr int tW1 = 18432;                          // W1 [c][u]: logits B (16 rows)
  static constexpr int tW1T = 20480;                         // W1^T [u][c]: input-gradient A (K = 16 classes)
  static constexpr int tDz = 0;                              // dz1 [b][c]: input-gradient B (K = 16 classes)
  static_assert(!kTCH || (kUPC == 64 && tW1T + 64 * 128 <= kFRing && tDzT + 16 * 128 <= tW1),
                "the head's operand tiles fit the F ring");
  static_assert(!kTCH || tW1 >= kZBytes, "the head-column tiles, written during the pair wait, clear the own partials");
  static_assert(2 * kW1Items * 16 <= kStagesF * B * kFBK * 2, "head-update partials must fit the F ring");
  // shared memory carve-up (bytes, from a 1024-aligned base)
  static constexpr int oRegion = 0;
  static constexpr int oW0 = (oRegion + kRegion + 1023) / 1024 * 1024;
  static constexpr int oDzT = oW0 + kMaxKb * kW0Blk;
  // the float h tile (CUDA-core last layer), which also receives the
  // partner's partials; with the tensor-core last layer only the latter
  static constexpr int kHsBytes = kTCH ? kZBytes : B * kHsd * 4;
  static constexpr int oHs = oDzT + kDzT;                    // [B][kHsd] float
  static constexpr int oWc = oHs + kHsBytes;                 // [C][kUPC] float (bf16 operand)
  static constexpr int oW1m = oWc + kFC * kUPC * 4;          // [C][kUPC] fp32 master head columns
  static constexpr int oPl = oW1m + kFC * kUPC * 4;          // [2][B][C] partial logits by step parity
  static constexpr int oDz = oPl + 2 * B * kFC * 4;          // [B][C]
  static constexpr int oDzb = oDz + B * kFC * 4;             // [C][B] (class-major; CUDA-core last layer)
  static constexpr int oGbp = oDzb + (kTCH ? 0 : B * kFC * 4);   // [kChunks][kUPC] (CUDA-core last layer)
  static constexpr int oRowLoss = oGbp + (kTCH ? 0 : kChunks * kUPC * 4);   // [B]
  static constexpr int oB0 = oRowLoss + B * 4;               // [kFU] b0 of the group's units
  static constexpr int oB1 = oB0 + kFU * 4;                  // [16] head bias (private copy)
  static constexpr int oLab = oB1 + 16 * 4;                  // [B] int
  static constexpr int oBar = (oLab + B * 4 + 15) / 16 * 16;
  static constexpr int kBarBytes = 256;
  static constexpr int kSmem = oBar + kBarBytes + 1024;      // + alignment slack
  static_assert(S == 1 || kUPC * kZs * 4 <= kHsBytes, "the incoming partials must fit the h tile they alias");
  static_assert(S == 1 || kZBytes <= kFRing, "own partials must fit the F ring");
};

struct FusedArgs {
  const int32_t* tau;       // [W]
  const int32_t* order;     // [W] workers, cluster by cluster
  const int32_t* cl_first;  // [clusters + 1] cluster k runs order[cl_first[k] .. cl_first[k + 1])
  int W, n_clusters, D, H;
  int global_slot;
  float lr;
  const float* master;      // slab read before the first step (the global slot)
  float* master_w;          // slab written during the last step (slot w)
  int64_t slot_stride;
  int64_t offW0, offB0, offW1, offB1;
  const int32_t* labels;    // [max_tau][W][B]
  int max_tau;
  int* err;
  unsigned long long* phase_ts;   // [max_tau][4] phase start stamps of worker 0 (or null)
  float* loss_out;                // [W]
  int64_t* cursor;                // [W]
  const int64_t* shard_n;         // [W]
};

template <int B, int S>
__global__ void __launch_bounds__(kFT, 1) fused_mlp2_round_kernel(const __grid_constant__ CUtensorMap mX,
                                                                 const __grid_constant__ CUtensorMap mXT,
                                                                 const __grid_constant__ CUtensorMap mW0f,
                                                                 const __grid_constant__ CUtensorMap mRep32,
                                                                 const __grid_constant__ CUtensorMap mRep16,
                                                                 const __grid_constant__ FusedArgs a) {
  using Cfg = FCfg<B, S>;
  constexpr int UPC = Cfg::kUPC;
  extern __shared__ uint8_t fs_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(fs_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* dring = sm + Cfg::oRegion;                // X^T tiles of step D
  uint8_t* fring = dring + Cfg::kDRing;              // X tiles of step F
  float* zx = reinterpret_cast<float*>(fring);       // [kUPC][kZs] own partials (S = 2), after the F MMAs
  uint8_t* w0s = sm + Cfg::oW0;                      // resident bf16 W0 block
  uint8_t* dzT = sm + Cfg::oDzT;
  float* hs = reinterpret_cast<float*>(sm + Cfg::oHs);
  // [kUPC][kZs] partials that the partner computed for this CTA's units
  // (S = 2).  They alias hs: the partner stores them in its forward epilogue,
  // after this CTA has passed the last barrier of its previous step (hs is
  // read only before it), and they are read into registers before hs is
  // rewritten.
  float* zin = hs;
  float* wcs = reinterpret_cast<float*>(sm + Cfg::oWc);
  float* w1m = reinterpret_cast<float*>(sm + Cfg::oW1m);
  float* pl = reinterpret_cast<float*>(sm + Cfg::oPl);
  float* dz = reinterpret_cast<float*>(sm + Cfg::oDz);
  float* dzb = reinterpret_cast<float*>(sm + Cfg::oDzb);
  float* gbp = reinterpret_cast<float*>(sm + Cfg::oGbp);
  float* rowloss = reinterpret_cast<float*>(sm + Cfg::oRowLoss);
  float* b0m = reinterpret_cast<float*>(sm + Cfg::oB0);
  float* b1m = reinterpret_cast<float*>(sm + Cfg::oB1);
  int* labs = reinterpret_cast<int*>(sm + Cfg::oLab);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + Cfg::oBar);
  uint64_t* fullF = bars;                      // [kStagesF]
  uint64_t* emptyF = fullF + Cfg::kStagesF;    // [kStagesF]
  uint64_t* accF = emptyF + Cfg::kStagesF;     // [1]
  uint64_t* fullD = accF + 1;                  // [kNXD] X^T tile landed
  uint64_t* xfreeD = fullD + kNXD;             // [kNXD] X^T tile consumed by its MMA
  uint64_t* accD = xfreeD + kNXD;              // [kNBD] TMEM buffer full
  uint64_t* pinF = accD + kNBD;                // [1] the partner's partials landed (S = 2)
  uint64_t* dzin = pinF + 1;                   // [1] the partner's dz0^T rows landed (S = 2)
  uint64_t* accH1 = dzin + 1;                  // [1] partial logits (tensor-core head)
  uint64_t* accH2 = accH1 + 1;                 // [1] input gradient and head-weight gradient (tensor-core head)
  uint64_t* ldW = accH2 + 1;                   // [1] model tiles landed (prologue)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(ldW + 1);

  const int rank = static_cast<int>(cluster_ctarank());
  const int ncl = static_cast<int>(gridDim.y);
  const int grp = rank / S, half = rank % S;    // unit group, column half
  const int g0 = grp * kFU;                     // first unit of the group
  const int ku0 = half * UPC;                   // first kept unit within the group
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int D = a.D, H = a.H;
  const int nkF = (D + kFBK - 1) / kFBK;
  const int kb_split = S > 1 ? nkF / 2 : nkF;
  const int kb_begin = half == 0 ? 0 : kb_split, kb_end = half == 0 ? kb_split : nkF;
  const int col_begin = kb_begin * kFBK;
  const int col_end = half == S - 1 ? D : kb_end * kFBK;
  const int ncols = col_end - col_begin;        // a multiple of 8
  const int nkf = kb_end - kb_begin;
  const int nD = (ncols + kND - 1) / kND;        // 32-column model tiles (load)
  const int nT = (ncols + kDT - 1) / kDT;        // 48-column weight-gradient tiles
  const int ncols16 = (ncols + 15) & ~15;        // columns the weight-gradient epilogue updates
  const int pre_f = nkf < Cfg::kStagesF ? nkf : Cfg::kStagesF;   // X tiles loaded ahead of a step
  const int pre_d = nT < kNXD ? nT : kNXD;                       // X^T tiles loaded before step D
  const int64_t gso = static_cast<int64_t>(a.global_slot) * a.slot_stride;
  const int partner = grp * S + (half ^ 1);     // S = 2: the other CTA of the group

  if (t == 0) {
    prefetch_tmap(&mX);
    prefetch_tmap(&mXT);
    prefetch_tmap(&mW0f);
    prefetch_tmap(&mRep32);
    prefetch_tmap(&mRep16);
    for (int i = 0; i < Cfg::kStagesF; ++i) {
      mbar_init(&fullF[i], 1);
      mbar_init(&emptyF[i], 1);
    }
    mbar_init(accF, 1);
    for (int i = 0; i < kNXD; ++i) {
      mbar_init(&fullD[i], 1);
      mbar_init(&xfreeD[i], 1);
    }
    for (int i = 0; i < kNBD; ++i) mbar_init(&accD[i], 1);
    mbar_init(pinF, 1);
    mbar_init(dzin, 1);
    mbar_init(accH1, 1);
    mbar_init(accH2, 1);
    mbar_init(ldW, 1);
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  // thread 0: fp32 tiles [tb, tb + kMaxKb) of the global model's W0 block
  // (the same for every worker of the cluster) by TMA into the
  // resident-operand area, completing on ldW.  Columns past D are zero (TMA
  // fill); every byte of the area that the tensor core reads later comes by
  // TMA or from the weight-gradient epilogue, so it needs no clearing.
  auto issue_w0f = [&](int tb) {
    const int nb = nD - tb < kMaxKb ? nD - tb : kMaxKb;
    mbar_arrive_expect_tx(ldW, nb * kW0Blk);   // an fp32 tile has the size of a bf16 K-block
    for (int i = 0; i < nb; ++i) tma_load_3d(w0s + i * kW0Blk, &mW0f, col_begin + (tb + i) * kND, g0, 0, ldW);
  };
  if (t == 0) issue_w0f(0);   // the first worker's first tiles are in flight during the set-up
  if (warp == 2) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  // zero the dz0^T tile (its K padding must stay zero for B < 64)
  for (int i = t; i < Cfg::kDzT / 16; i += kFT) reinterpret_cast<uint4*>(dzT)[i] = make_uint4(0, 0, 0, 0);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // every CTA's barriers are initialised before a peer signals them: the
  // arrival here, the wait before the first step
  if (S > 1) cluster_arrive();
  bool producer_ok = true;
  bool chain_ok = true;    // warps 1 and 3: no wait of this chain has run out
  int chain_tiles = 0;     // warps 1 and 3: tiles issued by this chain so far
  int sg0 = 0;             // steps this cluster ran for its earlier workers
  int ld_phase = 0;        // completed phases of ldW

  // The cluster's workers, one after the other (when there are more workers
  // than clusters that fit on the GPU, the host deals them longest first to
  // the cluster that will be free first).  Ring positions and barrier phases
  // follow the cluster's running step sg = sg0 + s; the staged inputs are
  // addressed by the worker and its own step s.
  for (int wi = a.cl_first[blockIdx.x]; wi < a.cl_first[blockIdx.x + 1]; ++wi) {
    const int w = a.order[wi];
    const int tau = a.tau[w];
    const int64_t dof = static_cast<int64_t>(w) * a.slot_stride;
    const bool stamp = a.phase_ts && w == 0 && rank == 0 && t == 0;

    // producer (warp 0 lane 0): X tiles [from, to) of step s's forward; the
    // ring position of K-block kb of step s is (sg0 + s) * nkf + kb
    auto issue_f = [&](int s, int from, int to) -> bool {
      for (int kb = from; kb < to; ++kb) {
        const int c = (sg0 + s) * nkf + kb, st = c % Cfg::kStagesF;
        if (c >= Cfg::kStagesF && !mbar_wait(&emptyF[st], ((c / Cfg::kStagesF) + 1) & 1, a.err, kDevTimeoutEmpty))
          return false;
        mbar_arrive_expect_tx(&fullF[st], Cfg::kBBytes);
        tma_load_4d(fring + st * Cfg::kBBytes, &mX, (kb_begin + kb) * kFBK, 0, w, s, &fullF[st]);
      }
      return true;
    };
    // X^T tiles [from, to) of step s's weight gradient (ring position (sg0 + s) * nT + tile)
    auto issue_d = [&](int s, int from, int to) -> bool {
      for (int tt = from; tt < to; ++tt) {
        const int c = (sg0 + s) * nT + tt, xb = c % kNXD, use = c / kNXD;
        // the buffer's previous tile must have been read by its MMA
        if (use >= 1 && !mbar_wait(&xfreeD[xb], (use - 1) & 1, a.err, kDevTimeoutEmpty)) return false;
        mbar_arrive_expect_tx(&fullD[xb], Cfg::kXtBytes);
        tma_load_4d(dring + xb * Cfg::kXtBytes, &mXT, 0, col_begin + tt * kDT, w, s, &fullD[xb]);
      }
      return true;
    };
    double loss_sum = 0.0;   // rank 0, thread 0: sum of the 16-row loss chunks, in step and chunk order

    // the global model, once per worker.  Warps 0-3: head columns and
    // biases.  The fp32 master block comes by TMA in tiles of 128 rows x 32
    // columns, up to kMaxKb at a time, into the resident-operand area (not in
    // use yet); the epilogue warps move each row to TMEM.  Then they write the
    // bf16 operand, rounded from the master in TMEM.  Columns past D are zero
    // (TMA fill).
    // the first X tiles of step 0 go out first (the F ring is free: the
    // previous worker's last forward has consumed it before the last barrier)
    if (warp == 0 && lane == 0) producer_ok = issue_f(0, 0, pre_f);
    if (warp < 4) {
      for (int q = t; q < kFC * (UPC / 4); q += 128) {
        const int c = q / (UPC / 4), u4 = (q % (UPC / 4)) * 4;
        const float4 m = *reinterpret_cast<const float4*>(a.master + gso + a.offW1 + static_cast<int64_t>(c) * H + g0 +
                                                         ku0 + u4);
        *reinterpret_cast<float4*>(w1m + c * UPC + u4) = m;
        *reinterpret_cast<float4*>(wcs + c * UPC + u4) =
            make_float4(bf16_round(m.x), bf16_round(m.y), bf16_round(m.z), bf16_round(m.w));
      }
      for (int u = t; u < kFU; u += 128) b0m[u] = a.master[gso + a.offB0 + g0 + u];
      if (t < kFC) b1m[t] = a.master[gso + a.offB1 + t];
    }
    for (int tb = 0; tb < nD; tb += kMaxKb) {
      const int nb = nD - tb < kMaxKb ? nD - tb : kMaxKb;
      if (t == 0 && (tb > 0 || wi != a.cl_first[blockIdx.x])) issue_w0f(tb);
      if (warp >= 4) {
        const int quarter = warp & 3, eg = (warp - 4) >> 2;
        const int r = quarter * 32 + lane;
        const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
        mbar_wait(ldW, ld_phase & 1, a.err, kDevTimeoutFull);
        for (int i = eg; i < nb; i += 2) {
          // row r of the tile: 128 bytes, 16-byte chunk q at (q ^ (r & 7))
          const uint8_t* row = w0s + i * kW0Blk + r * 128;
          float v[32];
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const float4 x = *reinterpret_cast<const float4*>(row + ((q ^ (r & 7)) << 4));
            v[4 * q] = x.x;
            v[4 * q + 1] = x.y;
            v[4 * q + 2] = x.z;
            v[4 * q + 3] = x.w;
          }
          tmem_st_32x32b_x32(trow + (tb + i) * kND, v);
        }
        tmem_wait_st();
      }
      ++ld_phase;
      tc_fence_before();
      __syncthreads();   // the tiles have been read before the area is written again
      tc_fence_after();
    }
    // the bf16 operand: the round-to-nearest bf16 of the fp32 master just
    // stored (the global model), K-block by K-block from TMEM into the
    // resident-operand area; columns past the CTA's last 32-column tile are
    // zero
    if (warp >= 4) {
      const int quarter = warp & 3, eg = (warp - 4) >> 2;
      const int r = quarter * 32 + lane;
      const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
      for (int j = eg; j < nkf; j += 2) {   // 2j < nD always
        float v0[32], v1[32];
        if (2 * j + 1 < nD) {
          tmem_ld_32x32b_x32_pair(trow + 2 * j * kND, v0, trow + (2 * j + 1) * kND, v1);
        } else {
          tmem_ld_32x32b_x32(trow + 2 * j * kND, v0);
#pragma unroll
          for (int i = 0; i < 32; ++i) v1[i] = 0.f;
        }
        put_w0_cols<32>(w0s, r, j * kFBK, v0);
        put_w0_cols<32>(w0s, r, j * kFBK + 32, v1);
      }
    }
    fence_proxy_async_smem();   // the resident W0 is read by the tensor core
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (S > 1 && wi == a.cl_first[blockIdx.x]) cluster_wait();

    for (int s = 0; s < tau; ++s) {
      if (stamp) a.phase_ts[s * 4 + 0] = global_ns();
      const bool last = s == tau - 1;
      const int sg = sg0 + s;
      if (S > 1 && t == 0) {   // what the partner sends this step: its partials and its dz0^T rows
        mbar_arrive_expect_tx(pinF, Cfg::kZTx);
        mbar_arrive_expect_tx(dzin, Cfg::kDzTx);
      }

      // ------------------------------------------------------------ F: partial forward of the group's units
      if (warp == 0 && lane == 0) {
        if (producer_ok) producer_ok = issue_f(s, pre_f, nkf);   // the rest of this step's X tiles
        if (producer_ok) producer_ok = issue_d(s, 0, pre_d);     // the first X^T tiles of step D
      } else if (warp == 1 && lane == 0) {
        constexpr uint32_t idesc = idesc_bf16_f32(128, B);
        for (int kb = 0; kb < nkf; ++kb) {
          const int c = sg * nkf + kb, st = c % Cfg::kStagesF;
          if (!mbar_wait(&fullF[st], (c / Cfg::kStagesF) & 1, a.err, kDevTimeoutFull)) break;
          tc_fence_after();
          const uint32_t wa = smem_u32(w0s + kb * kW0Blk);
          const uint32_t xb = smem_u32(fring + st * Cfg::kBBytes);
          // K slices of 16 wholly past the input's end (zero in both
          // operands) are not issued
          const int kleft = D - (kb_begin + kb) * kFBK;
#pragma unroll
          for (int j = 0; j < kFBK / 16; ++j)
            if (j * 16 < kleft)
              umma_bf16(tmem + kTAcc, smem_desc_k128(wa + j * 32), smem_desc_k128(xb + j * 32), idesc,
                        (kb | j) != 0 ? 1u : 0u);
          umma_commit(&emptyF[st]);
        }
        umma_commit(accF);
      }
      for (int b = t; b < B; b += kFT) labs[b] = a.labels[(static_cast<int64_t>(s) * a.W + w) * B + b];
      if (warp >= 4) {   // epilogue F: thread = unit of the group, columns = samples
        int ok = mbar_wait(accF, sg & 1, a.err, kDevTimeoutAccum) ? 1 : 0;
        ok = __all_sync(0xffffffffu, ok);
        tc_fence_after();
        if (ok) {
          const int quarter = warp & 3, eg = (warp - 4) >> 2;
          const int u = quarter * 32 + lane;
          const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + kTAcc;
          for (int c0 = eg * 32; c0 < B; c0 += 64) {
            float v[32];
            tmem_ld_32x32b_x32(trow + c0, v);
            if (S == 1) {
              const float bias = b0m[u];
#pragma unroll
              for (int j = 0; j < 32; ++j) hs[(c0 + j) * Cfg::kHsd + u] = bf16_round(fmaxf(v[j] + bias, 0.f));
            } else {
              // the partial goes to the CTA that keeps unit u: this one
              // (own rows) or the partner (its incoming buffer)
              const int owner = u / UPC;
              const int off = (u - owner * UPC) * Cfg::kZs + c0;
              if (owner == half) {
#pragma unroll
                for (int q = 0; q < 8; ++q)
                  *reinterpret_cast<float4*>(zx + off + 4 * q) =
                      make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
              } else {   // 16-byte asynchronous stores, counted on the partner's barrier
                const uint32_t dst = cluster_addr(zin + off, partner), bar = cluster_addr(pinF, partner);
#pragma unroll
                for (int q = 0; q < 8; ++q)
                  st_async_v4(dst + 16 * q, make_uint4(__float_as_uint(v[4 * q]), __float_as_uint(v[4 * q + 1]),
                                                       __float_as_uint(v[4 * q + 2]), __float_as_uint(v[4 * q + 3])),
                              bar);
              }
            }
          }
        }
      }
      tc_fence_before();
      __syncthreads();
      if (S > 1) {
        if constexpr (Cfg::kTCH) {
          // while the partner's partials are on their way: this CTA's head
          // columns (bf16 values) as the tensor core reads them, W1 [c][u]
          // (rows c < 10) and W1^T [u][c] (classes 10..15 zero: they multiply
          // the zero classes of dz1), clear of the own partials in the F ring
          for (int it = t; it < kFC * (UPC / 8) + UPC * 2; it += kFT) {
            if (it < kFC * (UPC / 8)) {
              const int c = it / (UPC / 8), u8 = (it % (UPC / 8)) * 8;
              const float* w = wcs + c * UPC + u8;
              *reinterpret_cast<uint4*>(fring + Cfg::tW1 + sw128_offset(c, u8)) =
                  make_uint4(pack_bf16x2(w[0], w[1]), pack_bf16x2(w[2], w[3]), pack_bf16x2(w[4], w[5]),
                             pack_bf16x2(w[6], w[7]));
            } else {
              const int i2 = it - kFC * (UPC / 8), u = i2 >> 1, c8 = (i2 & 1) * 8;
              float w[8];
#pragma unroll
              for (int i = 0; i < 8; ++i) w[i] = c8 + i < kFC ? wcs[(c8 + i) * UPC + u] : 0.f;
              *reinterpret_cast<uint4*>(fring + Cfg::tW1T + sw128_offset(u, c8)) =
                  make_uint4(pack_bf16x2(w[0], w[1]), pack_bf16x2(w[2], w[3]), pack_bf16x2(w[4], w[5]),
                             pack_bf16x2(w[6], w[7]));
            }
          }
        }
        // both partials of this CTA's units are local once the partner's
        // stores have landed:
        // z = part(half 0) + part(half 1) + b0
        mbar_wait(pinF, sg & 1, a.err, kDevTimeoutFull);
        constexpr int kZItems = UPC * (B / 4), kZPer = (kZItems + kFT - 1) / kFT;
        float4 zr[kZPer];
#pragma unroll
        for (int k = 0; k < kZPer; ++k) {
          const int q = t + k * kFT;
          if (q < kZItems) {   // item = (unit, 4 samples), consecutive threads on consecutive units
            const int ul = q % UPC, b4 = (q / UPC) * 4;
            const float4 own = *reinterpret_cast<const float4*>(zx + ul * Cfg::kZs + b4);
            const float4 inc = *reinterpret_cast<const float4*>(zin + ul * Cfg::kZs + b4);
            const float4 p0 = half == 0 ? own : inc, p1 = half == 0 ? inc : own;
            float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
            z.x += p0.x;
            z.y += p0.y;
            z.z += p0.z;
            z.w += p0.w;
            z.x += p1.x;
            z.y += p1.y;
            z.z += p1.z;
            z.w += p1.w;
            zr[k] = z;
          }
        }
        __syncthreads();   // the incoming partials (aliasing hs) have been read
#pragma unroll
        for (int k = 0; k < kZPer; ++k) {
          const int q = t + k * kFT;
          if (q >= kZItems) break;
          const int ul = q % UPC, b4 = (q / UPC) * 4;
          const int ug = ku0 + ul;                   // unit within the group
          const float4 z = zr[k];
          const float bias = b0m[ug];
          const float h0 = bf16_round(fmaxf(z.x + bias, 0.f)), h1 = bf16_round(fmaxf(z.y + bias, 0.f));
          const float h2 = bf16_round(fmaxf(z.z + bias, 0.f)), h3 = bf16_round(fmaxf(z.w + bias, 0.f));
          if constexpr (!Cfg::kTCH) {
            hs[(b4 + 0) * Cfg::kHsd + ul] = h0;
            hs[(b4 + 1) * Cfg::kHsd + ul] = h1;
            hs[(b4 + 2) * Cfg::kHsd + ul] = h2;
            hs[(b4 + 3) * Cfg::kHsd + ul] = h3;
          } else {   // h as the tensor core reads it, both ways (the only copy)
            st_bf16(fring + Cfg::tH + sw128_offset(b4 + 0, ul), h0);
            st_bf16(fring + Cfg::tH + sw128_offset(b4 + 1, ul), h1);
            st_bf16(fring + Cfg::tH + sw128_offset(b4 + 2, ul), h2);
            st_bf16(fring + Cfg::tH + sw128_offset(b4 + 3, ul), h3);
            *reinterpret_cast<uint2*>(fring + Cfg::tHT + sw128_offset(ul, b4)) =
                make_uint2(pack_bf16x2(h0, h1), pack_bf16x2(h2, h3));
          }
        }
        if constexpr (Cfg::kTCH) fence_proxy_async_smem();   // the h tiles are read by the tensor core
        __syncthreads();
      }
      if (stamp) a.phase_ts[s * 4 + 1] = global_ns();

      // ------------------------------------------------------------ H: last layer for this CTA's units
      float* plb = pl + (sg & 1) * B * kFC;   // this step's partial logits (read by every CTA)
      if constexpr (Cfg::kTCH) {
        // partial logits plb[b][c] = sum over this CTA's units of h[b][u] W1[c][u]:
        // M = 128 (rows b < 64 used), N = 16 (classes < 10 used), K = 64 units
        if (warp == 1 && lane == 0) {
          tc_fence_after();
          constexpr uint32_t idesc = idesc_bf16_f32(128, 16);
          const uint32_t ha = smem_u32(fring + Cfg::tH), wb = smem_u32(fring + Cfg::tW1);
#pragma unroll
          for (int j = 0; j < kFBK / 16; ++j)
            umma_bf16(tmem + kTAcc + 64, smem_desc_k128(ha + j * 32), smem_desc_k128(wb + j * 32), idesc, j != 0 ? 1u : 0u);
          umma_commit(accH1);
        } else if (warp == 4 || warp == 5) {   // lanes 0..63: one sample each
          int ok = mbar_wait(accH1, sg & 1, a.err, kDevTimeoutAccum) ? 1 : 0;
          ok = __all_sync(0xffffffffu, ok);
          tc_fence_after();
          if (ok) {
            float v[16];
            tmem_ld_32x32b_x16(tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16) + kTAcc + 64, v);
            const int b = (warp & 3) * 32 + lane;
#pragma unroll
            for (int c = 0; c < kFC; ++c) plb[b * kFC + c] = v[c];
          }
          tc_fence_before();
        }
      } else if (t < 256) {   // partial logits: kTpr threads per row, all classes in registers
        const int rb = t / Cfg::kTpr, q = t % Cfg::kTpr;
        float acc[kFC];
#pragma unroll
        for (int c = 0; c < kFC; ++c) acc[c] = 0.f;
        for (int k = 4 * q; k < UPC; k += 4 * Cfg::kTpr) {
          const float4 hv = *reinterpret_cast<const float4*>(hs + rb * Cfg::kHsd + k);
#pragma unroll
          for (int c = 0; c < kFC; ++c) {
            const float4 wv = *reinterpret_cast<const float4*>(wcs + c * UPC + k);
            acc[c] = fmaf(hv.x, wv.x, acc[c]);
            acc[c] = fmaf(hv.y, wv.y, acc[c]);
            acc[c] = fmaf(hv.z, wv.z, acc[c]);
            acc[c] = fmaf(hv.w, wv.w, acc[c]);
          }
        }
#pragma unroll
        for (int c = 0; c < kFC; ++c) {
          for (int o = Cfg::kTpr / 2; o > 0; o >>= 1) acc[c] += __shfl_xor_sync(0xffffffffu, acc[c], o);
          if (q == 0) plb[rb * kFC + c] = acc[c];
        }
      }
      cluster_sync();
      // logits: the partials of every CTA of the cluster in rank order, then
      // the bias; four consecutive logits per thread (16-byte remote loads)
      static_assert((B * kFC) % 4 == 0 && (Cfg::oPl % 16) == 0, "16-byte items of the partial logits");
      for (int q4 = t; q4 < B * kFC / 4; q4 += kFT) {
        float4 part[kFMaxCluster];
#pragma unroll
        for (int r = 0; r < kFMaxCluster; ++r)
          part[r] = r < ncl ? ld_dsmem_f32x4(plb + 4 * q4, r) : make_float4(0.f, 0.f, 0.f, 0.f);
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int r = 0; r < kFMaxCluster; ++r)
          if (r < ncl) {
            acc.x += part[r].x;
            acc.y += part[r].y;
            acc.z += part[r].z;
            acc.w += part[r].w;
          }
        const int q = 4 * q4;
        dz[q] = acc.x + b1m[q % kFC];
        dz[q + 1] = acc.y + b1m[(q + 1) % kFC];
        dz[q + 2] = acc.z + b1m[(q + 2) % kFC];
        dz[q + 3] = acc.w + b1m[(q + 3) % kFC];
      }
      __syncthreads();   // the softmax rows below read logits summed by other threads
      // softmax cross-entropy, four threads per row: thread q of the row takes
      // classes q, q + 4, q + 8 (exponentials and gradients); the row's
      // exponentials are gathered in every lane of the row and summed in class
      // order (the arithmetic of one thread per row)
      static_assert(4 * B <= kFT, "four threads per batch row");
      if (t < 4 * B) {
        const int b = t >> 2, q = t & 3, src = lane & ~3;
        float zq[3], eq[3];
#pragma unroll
        for (int i = 0; i < 3; ++i) zq[i] = q + 4 * i < kFC ? dz[b * kFC + q + 4 * i] : -INFINITY;
        float m = fmaxf(fmaxf(zq[0], zq[1]), zq[2]);
        m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 1));
        m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 2));
#pragma unroll
        for (int i = 0; i < 3; ++i) eq[i] = q + 4 * i < kFC ? expf(zq[i] - m) : 0.f;
        const int y = labs[b];
        float se = 0.f, so_ = 0.f;
#pragma unroll
        for (int c = 0; c < kFC; ++c) {
          const float ec = __shfl_sync(0xffffffffu, eq[c >> 2], src | (c & 3));
          se += ec;
          if (c != y) so_ += ec;
        }
        if (q == (y & 3)) rowloss[b] = m + logf(se) - (y < 4 ? zq[0] : y < 8 ? zq[1] : zq[2]);
        const float inv = 1.0f / static_cast<float>(B);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int c = q + 4 * i;
          if (i < 3 && c < kFC) {
            const float g = (c == y ? -(so_ / se) : eq[i < 3 ? i : 2] / se) * inv;
            dz[b * kFC + c] = g;
            if constexpr (Cfg::kTCH) {   // dz1 as the tensor core reads it, both ways
              st_bf16(fring + Cfg::tDz + sw128_offset(b, c), g);
              st_bf16(fring + Cfg::tDzT + sw128_offset(c, b), g);
            } else {
              dzb[c * B + b] = bf16_round(g);
            }
          } else if (Cfg::kTCH) {
            st_bf16(fring + Cfg::tDz + sw128_offset(b, c), 0.f);   // classes 10..15 of the K = 16 operand
          }
        }
      }
      if constexpr (Cfg::kTCH) fence_proxy_async_smem();   // the dz1 tiles are read by the tensor core
      tc_fence_before();
      __syncthreads();
      tc_fence_after();
      if (rank == 0 && t == 0) {
        for (int c = 0; c < B / kRowsPerLossChunk; ++c) {
          float l = 0.f;
          for (int r = 0; r < kRowsPerLossChunk; ++r) l += rowloss[c * kRowsPerLossChunk + r];
          loss_sum += static_cast<double>(l);
        }
      }
      if (warp >= 8 && warp < 11) {   // head bias, 8 lanes per class: the same arithmetic in every CTA
        const int idx = t - 256, c = idx >> 3, j = idx & 7;
        float g = 0.f;
        if (c < kFC)
          for (int b = j; b < B; b += 8) g += dz[b * kFC + c];
#pragma unroll
        for (int o = 4; o > 0; o >>= 1) g += __shfl_xor_sync(0xffffffffu, g, o, 8);
        if (j == 0 && c < kFC) {
          const float nb = fmaf(-a.lr, g, b1m[c]);
          b1m[c] = nb;
          if (last && rank == 0) a.master_w[dof + a.offB1 + c] = nb;
        }
      }
      if constexpr (Cfg::kTCH) {
        // the input gradient dh^T[u][b] = sum_c W1^T[u][c] dz1[b][c] (M = 128
        // with rows u < 64 used, N = 64 samples, K = 16 classes) and the
        // head-weight gradient dW1^T[u][c] = sum_b h^T[u][b] dz1^T[c][b]
        // (N = 16 with classes < 10 used, K = 64 samples), one commit
        if (warp == 1 && lane == 0) {
          umma_bf16(tmem + kTAcc, smem_desc_k128(smem_u32(fring + Cfg::tW1T)), smem_desc_k128(smem_u32(fring + Cfg::tDz)),
                    idesc_bf16_f32(128, B), 0u);
          constexpr uint32_t idesc = idesc_bf16_f32(128, 16);
          const uint32_t ha = smem_u32(fring + Cfg::tHT), gb = smem_u32(fring + Cfg::tDzT);
#pragma unroll
          for (int j = 0; j < kFBK / 16; ++j)
            umma_bf16(tmem + kTAcc + 64, smem_desc_k128(ha + j * 32), smem_desc_k128(gb + j * 32), idesc, j != 0 ? 1u : 0u);
          umma_commit(accH2);
        } else if (warp == 4 || warp == 5) {
          // unit u = (warp & 3) * 32 + lane: its masked dz0 row (bf16 into the
          // K-major dz0^T tile, the A operand of step D) and its b0 (the sum
          // of the fp32 masked gradient)
          int ok = mbar_wait(accH2, sg & 1, a.err, kDevTimeoutAccum) ? 1 : 0;
          ok = __all_sync(0xffffffffu, ok);
          tc_fence_after();
          const int u = (warp & 3) * 32 + lane;
          const uint32_t trow = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16) + kTAcc;
          float gsum = 0.f;
          if (ok) {
            for (int c0 = 0; c0 < B; c0 += 32) {
              float v[32];
              tmem_ld_32x32b_x32(trow + c0, v);
              // ReLU mask from unit u's row of the bf16 h^T tile: h >= 0, so
              // h > 0 exactly when its bf16 bits are not zero
              uint32_t hb[16];
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                const uint4 q = *reinterpret_cast<const uint4*>(fring + Cfg::tHT + sw128_offset(u, c0 + 8 * k));
                hb[4 * k] = q.x;
                hb[4 * k + 1] = q.y;
                hb[4 * k + 2] = q.z;
                hb[4 * k + 3] = q.w;
              }
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                const uint32_t bits = (hb[i >> 1] >> ((i & 1) * 16)) & 0xFFFFu;
                const float dh = bits != 0u ? v[i] : 0.f;
                v[i] = dh;
                gsum += dh;
              }
#pragma unroll
              for (int k = 0; k < 4; ++k)
                *reinterpret_cast<uint4*>(dzT + sw128_offset(ku0 + u, c0 + 8 * k)) =
                    make_uint4(pack_bf16x2(v[8 * k], v[8 * k + 1]), pack_bf16x2(v[8 * k + 2], v[8 * k + 3]),
                               pack_bf16x2(v[8 * k + 4], v[8 * k + 5]), pack_bf16x2(v[8 * k + 6], v[8 * k + 7]));
            }
          }
          const float nb = fmaf(-a.lr, gsum, b0m[ku0 + u]);
          b0m[ku0 + u] = nb;
          if (last) a.master_w[dof + a.offB0 + g0 + ku0 + u] = nb;
          tc_fence_before();
        } else if (warp == 8 || warp == 9) {
          // SGD of the head-weight column of unit u = (warp & 3) * 32 + lane
          int ok = mbar_wait(accH2, sg & 1, a.err, kDevTimeoutAccum) ? 1 : 0;
          ok = __all_sync(0xffffffffu, ok);
          tc_fence_after();
          const int u = (warp & 3) * 32 + lane;
          if (ok) {
            float v[16];
            tmem_ld_32x32b_x16(tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16) + kTAcc + 64, v);
#pragma unroll
            for (int c = 0; c < kFC; ++c) {
              const float nw = fmaf(-a.lr, v[c], w1m[c * UPC + u]);
              w1m[c * UPC + u] = nw;
              wcs[c * UPC + u] = bf16_round(nw);
              if (last) a.master_w[dof + a.offW1 + static_cast<int64_t>(c) * H + g0 + ku0 + u] = nw;
            }
          }
          tc_fence_before();
        }
        fence_proxy_async_smem();   // dz0^T is read by the tensor core next
        __syncthreads();
      if (S > 1) {   // h is not read again this step: this CTA's dz0^T rows to the partner
        const uint32_t dst = cluster_addr(dzT, partner), bar = cluster_addr(dzin, partner);
        for (int it = t; it < UPC * Cfg::kChunks; it += kFT) {
          const uint32_t off = sw128_offset(ku0 + it / Cfg::kChunks, 8 * (it % Cfg::kChunks));
          st_async_v4(dst + off, *reinterpret_cast<const uint4*>(dzT + off), bar);
        }
      }
      } else {
        // masked input gradient dz0[b][u] of this CTA's units: item = (unit, 8
        // consecutive samples), one 16-byte chunk of the unit's K-major dz0^T
        // row
        for (int it = t; it < UPC * Cfg::kChunks; it += kFT) {
          const int u = it % UPC, j = it / UPC;
          // dh[b] = sum over c in class order of dzb[c][b] w[c][u]: the eight
          // samples of a class are two 16-byte loads of the class-major dzb
          float dv[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) dv[i] = 0.f;
#pragma unroll
          for (int c = 0; c < kFC; ++c) {
            const float wc = wcs[c * UPC + u];
            const float4 d0 = *reinterpret_cast<const float4*>(dzb + c * B + 8 * j);
            const float4 d1 = *reinterpret_cast<const float4*>(dzb + c * B + 8 * j + 4);
            dv[0] = fmaf(d0.x, wc, dv[0]);
            dv[1] = fmaf(d0.y, wc, dv[1]);
            dv[2] = fmaf(d0.z, wc, dv[2]);
            dv[3] = fmaf(d0.w, wc, dv[3]);
            dv[4] = fmaf(d1.x, wc, dv[4]);
            dv[5] = fmaf(d1.y, wc, dv[5]);
            dv[6] = fmaf(d1.z, wc, dv[6]);
            dv[7] = fmaf(d1.w, wc, dv[7]);
          }
          float gsum = 0.f;
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const float dh = hs[(8 * j + i) * Cfg::kHsd + u] > 0.f ? dv[i] : 0.f;
            dv[i] = dh;
            gsum += dh;
          }
          const uint4 p = make_uint4(pack_bf16x2(dv[0], dv[1]), pack_bf16x2(dv[2], dv[3]), pack_bf16x2(dv[4], dv[5]),
                                     pack_bf16x2(dv[6], dv[7]));
          *reinterpret_cast<uint4*>(dzT + sw128_offset(ku0 + u, 8 * j)) = p;
          gbp[j * UPC + u] = gsum;
        }
        fence_proxy_async_smem();   // dz0^T is read by the tensor core next
        __syncthreads();
        // head weight gradient of this CTA's columns, item = (class, 4 units),
        // split over the two halves of the batch (partials in the idle F ring)
        float4* w1p = reinterpret_cast<float4*>(fring);   // [2][kW1Items]
        for (int q = t; q < 2 * Cfg::kW1Items; q += kFT) {
          const int item = q % Cfg::kW1Items, hb = q / Cfg::kW1Items;
          const int c = item / (UPC / 4), u4 = (item % (UPC / 4)) * 4;
          float4 dw = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 2
          for (int b4 = hb * (B / 2); b4 < (hb + 1) * (B / 2); b4 += 4) {
            const float4 g4 = *reinterpret_cast<const float4*>(dzb + c * B + b4);   // samples b4 .. b4 + 3
            const float gk[4] = {g4.x, g4.y, g4.z, g4.w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const float4 hv = *reinterpret_cast<const float4*>(hs + (b4 + k) * Cfg::kHsd + u4);
              dw.x = fmaf(gk[k], hv.x, dw.x);
              dw.y = fmaf(gk[k], hv.y, dw.y);
              dw.z = fmaf(gk[k], hv.z, dw.z);
              dw.w = fmaf(gk[k], hv.w, dw.w);
            }
          }
          w1p[hb * Cfg::kW1Items + item] = dw;
        }
        if (t < UPC) {   // b0 of this CTA's units (chunk sums in chunk order)
          float g = 0.f;
#pragma unroll
          for (int r = 0; r < Cfg::kChunks; ++r) g += gbp[r * UPC + t];
          const float nb = fmaf(-a.lr, g, b0m[ku0 + t]);
          b0m[ku0 + t] = nb;
          if (last) a.master_w[dof + a.offB0 + g0 + ku0 + t] = nb;
        }
        __syncthreads();
        if (S > 1) {   // h is not read again this step: this CTA's dz0^T rows to the partner
          const uint32_t dst = cluster_addr(dzT, partner), bar = cluster_addr(dzin, partner);
          for (int it = t; it < UPC * Cfg::kChunks; it += kFT) {
            const uint32_t off = sw128_offset(ku0 + it / Cfg::kChunks, 8 * (it % Cfg::kChunks));
            st_async_v4(dst + off, *reinterpret_cast<const uint4*>(dzT + off), bar);
          }
        }
        // SGD of the head-weight columns: first half + second half of the batch
        for (int item = t; item < Cfg::kW1Items; item += kFT) {
          const int c = item / (UPC / 4), u4 = (item % (UPC / 4)) * 4;
          const float4 d0 = w1p[item], d1 = w1p[Cfg::kW1Items + item];
          const float4 dw = make_float4(d0.x + d1.x, d0.y + d1.y, d0.z + d1.z, d0.w + d1.w);
          const float4 o = *reinterpret_cast<const float4*>(w1m + c * UPC + u4);
          float4 nw;
          nw.x = fmaf(-a.lr, dw.x, o.x);
          nw.y = fmaf(-a.lr, dw.y, o.y);
          nw.z = fmaf(-a.lr, dw.z, o.z);
          nw.w = fmaf(-a.lr, dw.w, o.w);
          *reinterpret_cast<float4*>(w1m + c * UPC + u4) = nw;
          *reinterpret_cast<float4*>(wcs + c * UPC + u4) =
              make_float4(bf16_round(nw.x), bf16_round(nw.y), bf16_round(nw.z), bf16_round(nw.w));
          if (last)
            *reinterpret_cast<float4*>(a.master_w + dof + a.offW1 + static_cast<int64_t>(c) * H + g0 + ku0 + u4) = nw;
        }
      }
      if (stamp) a.phase_ts[s * 4 + 2] = global_ns();

      // ------------------------------------------------------------ D: weight gradient + SGD of own W0 block
      if (warp == 0 && lane == 0) {
        if (producer_ok) producer_ok = issue_d(s, pre_d, nT);
        // the first X tiles of the next step's forward, while this step's epilogue runs
        if (producer_ok && s + 1 < tau) producer_ok = issue_f(s + 1, 0, pre_f);
      } else if (warp == 1 || warp == 3) {
        // two issuing chains: chain e (warp 1: e = 0, warp 3: e = 1) takes the
        // tiles with running index c = e (mod 2), TMEM buffer e, X^T slots
        // c % 4 (of its own parity) and epilogue warpgroup e.  The warpgroup
        // hands the drained buffer back through named barrier 1 + e (128
        // arrivals + this warp: cheaper than an mbarrier wait); every tile is
        // committed, even after a failed wait, so that the arrivals and the
        // waits on the named barrier stay paired
        const int e = warp == 1 ? 0 : 1;
        constexpr uint32_t idesc = idesc_bf16_f32(128, kDT);
        if (S > 1) {   // the partner's dz0^T rows (st.async) have landed before the tensor core reads them
          if (chain_ok) chain_ok = mbar_wait(dzin, sg & 1, a.err, kDevTimeoutFull);
          fence_proxy_async_smem();
        }
        for (int tt = ((sg * nT + e) & 1); tt < nT; tt += 2) {
          const int c = sg * nT + tt, buf = e, use = c / kNBD, xb = c % kNXD;
          if (chain_ok) chain_ok = mbar_wait(&fullD[xb], (c / kNXD) & 1, a.err, kDevTimeoutFull);
          if (use >= 1) bar_named(1 + e, 128 + 32);   // the previous use of the buffer has been read
          tc_fence_after();
          if (lane == 0) {
            if (chain_ok) {
              const uint32_t xa = smem_u32(dring + xb * Cfg::kXtBytes);
              const uint32_t da = smem_u32(dzT);
              const uint32_t dcol = tmem + static_cast<uint32_t>(kTAcc + buf * kDT);
#pragma unroll
              for (int j = 0; j < kFBK / 16; ++j)
                umma_bf16(dcol, smem_desc_k128(da + j * 32), smem_desc_k128(xa + j * 32), idesc, j != 0 ? 1u : 0u);
            }
            umma_commit(&accD[buf]);
            umma_commit(&xfreeD[xb]);
          }
          __syncwarp();
          ++chain_tiles;
        }
      } else if (warp >= 4) {
        // warpgroup eg drains the tiles of chain eg (its TMEM buffer); a warp
        // covers 32 rows
        const int quarter = warp & 3, eg = (warp - 4) >> 2;
        const int r = quarter * 32 + lane;
        const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
        // the last step's updated master goes to the worker's replica slot by
        // TMA stores from two staging buffers per warp in the resident-operand
        // area (not read again by this worker once the step's forward has
        // run): 32 columns as a 128-byte-swizzled 32 x 32 box, 16 columns as
        // a plain 32 x 16 box
        uint8_t* stg = w0s + (warp - 4) * kStgBytes;
        int nst = 0;   // tiles this warp has stored
        for (int tt = ((sg * nT + eg) & 1); tt < nT; tt += 2) {
          const int c = sg * nT + tt, buf = eg, use = c / kNBD;
          int ok = mbar_wait(&accD[buf], use & 1, a.err, kDevTimeoutAccum) ? 1 : 0;
          ok = __all_sync(0xffffffffu, ok);
          tc_fence_after();
          if (ok) {
            // the tile's columns up to the input's end rounded to 16 (the
            // padding columns past the input are zero in the master and in
            // X^T): 32 and/or 16 columns, the same for the whole warp
            const int c0 = tt * kDT;
            const int nc = ncols16 - c0 < kDT ? ncols16 - c0 : kDT;
            const bool has32 = nc >= 32, has16 = (nc & 16) != 0;
            const int c16 = c0 + (has32 ? 32 : 0);
            const uint32_t gcol = trow + kTAcc + buf * kDT;
            // the gradient first: once it is in registers the buffer goes back
            // to the issuing chain; the master columns are this thread's own
            float g[32], g16[16];
            if (has32) tmem_ld_32x32b_x32(gcol, g);
            if (has16) tmem_ld_32x32b_x16(gcol + (has32 ? 32 : 0), g16);
            tc_fence_before();
            bar_arrive_named(1 + eg, 128 + 32);   // the gradient buffer has been read: the next MMA may reuse it
            uint8_t* st32 = stg + (nst & 1) * kStg32;
            uint8_t* st16 = stg + 2 * kStg32 + (nst & 1) * kStg16;
            if (last) {   // the store of two tiles ago has read this buffer pair
              if (lane == 0 && nst >= 2) bulk_wait_read_but_one();
              __syncwarp();
            }
            if (has32) {
              float m[32];
              tmem_ld_32x32b_x32(trow + c0, m);
#pragma unroll
              for (int j = 0; j < 32; ++j) m[j] = fmaf(-a.lr, g[j], m[j]);
              if (!last) {
                tmem_st_32x32b_x32(trow + c0, m);
                put_w0_cols<32>(w0s, r, c0, m);
              } else {   // row `lane`: 16-byte chunk q at (q ^ (lane & 7))
#pragma unroll
                for (int q = 0; q < 8; ++q)
                  *reinterpret_cast<float4*>(st32 + lane * 128 + ((q ^ (lane & 7)) << 4)) =
                      make_float4(m[4 * q], m[4 * q + 1], m[4 * q + 2], m[4 * q + 3]);
              }
            }
            if (has16) {
              float m16[16];
              tmem_ld_32x32b_x16(trow + c16, m16);
#pragma unroll
              for (int j = 0; j < 16; ++j) m16[j] = fmaf(-a.lr, g16[j], m16[j]);
              if (!last) {
                tmem_st_32x32b_x16(trow + c16, m16);
                put_w0_cols<16>(w0s, r, c16, m16);
              } else {
#pragma unroll
                for (int q = 0; q < 4; ++q)
                  *reinterpret_cast<float4*>(st16 + lane * 64 + q * 16) =
                      make_float4(m16[4 * q], m16[4 * q + 1], m16[4 * q + 2], m16[4 * q + 3]);
              }
            }
            if (last) {
              fence_proxy_async_smem();   // the staged rows are read by the TMA store
              __syncwarp();
              if (lane == 0) {
                if (has32) tma_store_3d(&mRep32, st32, col_begin + c0, g0 + quarter * 32, w);
                if (has16) tma_store_3d(&mRep16, st16, col_begin + c16, g0 + quarter * 32, w);
                bulk_commit_group();
              }
              ++nst;
            }
          } else {
            tc_fence_before();
            bar_arrive_named(1 + eg, 128 + 32);
          }
        }
        tmem_wait_st();   // the master columns stored above are read again next step
        // the staging buffers are read before the next worker's model comes in
        if (last && lane == 0) bulk_wait_read_all();
      }
      fence_proxy_async_smem();   // the resident W0 written here is read by the tensor core next step
      tc_fence_before();
      __syncthreads();
      tc_fence_after();
      if (stamp) a.phase_ts[s * 4 + 3] = global_ns();
    }
    // round bookkeeping of this worker (its W0 block went to its replica slot
    // by TMA stores in the last step): mean loss over its steps and the data
    // cursor
    if (rank == 0 && t == 0) {
      a.loss_out[w] = static_cast<float>(loss_sum / (static_cast<double>(B) * tau));
      if (a.cursor) a.cursor[w] = (a.cursor[w] + static_cast<int64_t>(tau) * B) % a.shard_n[w];
    }
    // the last step has read TMEM before the next worker's model goes in
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    sg0 += tau;
  }
  // the last drain of each chain's buffer pairs with one more wait
  if ((warp == 1 || warp == 3) && chain_tiles > 0) bar_named(1 + (warp == 1 ? 0 : 1), 128 + 32);
  // every replica store has completed before the kernel ends
  if (warp >= 4 && lane == 0) bulk_wait_all();
  // (a cluster without workers still completes the set-up barrier)
  if (S > 1 && a.cl_first[blockIdx.x] == a.cl_first[blockIdx.x + 1]) cluster_wait();
  cluster_sync();   // peers may still read this CTA's partial logits of the last step
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int B, int S>
cudaError_t launch_bs(const CUtensorMap& mX, const CUtensorMap& mXT, const CUtensorMap& mW0f, const CUtensorMap& mRep32,
                      const CUtensorMap& mRep16, const FusedArgs& a, int priority, cudaStream_t s) {
  using Cfg = FCfg<B, S>;
  cudaError_t e = cudaFuncSetAttribute(fused_mlp2_round_kernel<B, S>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg::kSmem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.n_clusters, S * (a.H / kFU), 1);
  cfg.blockDim = dim3(kFT, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int n = 0;
  attr[n].id = cudaLaunchAttributeClusterDimension;
  attr[n].val.clusterDim.x = 1;
  attr[n].val.clusterDim.y = S * (a.H / kFU);
  attr[n].val.clusterDim.z = 1;
  ++n;
  if (priority != 0) {   // ahead of concurrent work (the next round's staging) for free SMs
    attr[n].id = cudaLaunchAttributePriority;
    attr[n].val.priority = priority;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, fused_mlp2_round_kernel<B, S>, mX, mXT, mW0f, mRep32, mRep16, a);
}

// two CTAs per unit group when the cluster stays within 8 CTAs and the input
// has at least two K-blocks
int split_for(int D, int H) { return (2 * (H / kFU) <= kFMaxCluster && (D + kFBK - 1) / kFBK >= 2) ? 2 : 1; }

// input columns of the widest CTA of a group (the last one)
int widest_cols(int D, int S) {
  const int nkF = (D + kFBK - 1) / kFBK;
  return S > 1 ? D - (nkF / 2) * kFBK : D;
}

}  // namespace

bool fused_round_supported(int L, int D, int H, int C, int B) {
  if (L != 2 || C != kFC || H % kFU != 0 || H / kFU > kFMaxCluster || D % 8 != 0) return false;
  if (B != 32 && B != 64) return false;
  const int S = split_for(D, H);
  // the CTA's master block must fit the TMEM columns below the accumulators
  if ((widest_cols(D, S) + kND - 1) / kND * kND > kTAcc) return false;
  int smem = 0;
  if (B == 32) smem = S == 2 ? FCfg<32, 2>::kSmem : FCfg<32, 1>::kSmem;
  else smem = S == 2 ? FCfg<64, 2>::kSmem : FCfg<64, 1>::kSmem;
  return smem <= 227 * 1024;
}

int fused_round_xt_rows(int) { return kDT; }

namespace {
template <int B, int S>
int max_clusters_bs(int H) {
  using Cfg = FCfg<B, S>;
  if (cudaFuncSetAttribute(fused_mlp2_round_kernel<B, S>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmem) !=
      cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  const int ncl = S * (H / kFU);
  cfg.gridDim = dim3(1, ncl, 1);
  cfg.blockDim = dim3(kFT, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmem;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = 1;
  attr.val.clusterDim.y = ncl;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, fused_mlp2_round_kernel<B, S>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}
}  // namespace

int fused_round_max_clusters(int D, int H, int B) {
  const int S = split_for(D, H);
  if (B == 32) return S == 2 ? max_clusters_bs<32, 2>(H) : max_clusters_bs<32, 1>(H);
  if (B == 64) return S == 2 ? max_clusters_bs<64, 2>(H) : max_clusters_bs<64, 1>(H);
  return 0;
}

cudaError_t launch_fused_round(const CUtensorMap& mX, const CUtensorMap& mXT, const CUtensorMap& mW0f,
                               const CUtensorMap& mRep32, const CUtensorMap& mRep16, const FusedRoundArgs& r,
                               cudaStream_t s) {
  FusedArgs a;
  a.tau = r.tau;
  a.order = r.order;
  a.cl_first = r.cl_first;
  a.W = r.W;
  a.n_clusters = r.n_clusters;
  a.D = r.D;
  a.H = r.H;
  a.global_slot = r.global_slot;
  a.lr = r.lr;
  a.master = r.master;
  a.master_w = r.master_w;
  a.slot_stride = r.slot_stride;
  a.offW0 = r.offW0;
  a.offB0 = r.offB0;
  a.offW1 = r.offW1;
  a.offB1 = r.offB1;
  a.labels = r.labels;
  a.max_tau = r.max_tau;
  a.err = r.err;
  a.phase_ts = r.phase_ts;
  a.loss_out = r.loss_out;
  a.cursor = r.cursor;
  a.shard_n = r.shard_n;
  const int S = split_for(r.D, r.H);
  if (r.B == 32)
    return S == 2 ? launch_bs<32, 2>(mX, mXT, mW0f, mRep32, mRep16, a, r.priority, s)
                  : launch_bs<32, 1>(mX, mXT, mW0f, mRep32, mRep16, a, r.priority, s);
  if (r.B == 64)
    return S == 2 ? launch_bs<64, 2>(mX, mXT, mW0f, mRep32, mRep16, a, r.priority, s)
                  : launch_bs<64, 1>(mX, mXT, mW0f, mRep32, mRep16, a, r.priority, s);
  return cudaErrorInvalidValue;
}

}  // namespace oscars
