// Measurement probes of bench.py (not part of libstepprune): the on-chip peaks
// the selection kernel's traffic is reported against (aggregate shared-memory
// and L2 read bandwidth), and the per-round floor of its cluster
// synchronisation (the round skeleton of the selection kernel -- two DSMEM push
// exchanges, two cluster barriers, the block reductions -- with no candidate or
// history work).  Each call allocates what it needs, runs on the current
// device, synchronises and returns the figure; the return value is the CUDA
// error code (0 = success).
//
//   nvcc -gencode arch=compute_103a,code=sm_103a -O3 -shared -Xcompiler -fPIC \
//        bench_probes.cu -o bench_probes.so       (bench.py's build_probes())
#include <cooperative_groups.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>

namespace cg = cooperative_groups;

namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

int sm_count() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n;
}

constexpr int PNT = 512;
constexpr int SMEM_F4 = 4096;  // 64 KB per CTA

__global__ void __launch_bounds__(PNT) smem_read_kernel(int iters, float* __restrict__ sink) {
  extern __shared__ float4 buf4[];
  for (int i = threadIdx.x; i < SMEM_F4; i += PNT) buf4[i] = make_float4((float)i, 1.f, 2.f, 3.f);
  __syncthreads();
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  int idx = threadIdx.x;
  const uint32_t base = smem_u32(buf4);
#pragma unroll 8
  for (int it = 0; it < iters; ++it) {
    float4 v;
    // volatile: every read is issued (the buffer does not change, so plain
    // loads of the repeating addresses could be merged)
    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(base + (uint32_t)idx * 16u));
    acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
    idx = (idx + PNT) & (SMEM_F4 - 1);
  }
  sink[blockIdx.x * PNT + threadIdx.x] = acc.x + acc.y + acc.z + acc.w;
}

__global__ void __launch_bounds__(PNT) l2_read_kernel(const float4* __restrict__ src, size_t n4, int passes,
                                                      float* __restrict__ sink) {
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  const size_t stride = (size_t)gridDim.x * PNT;
  for (int p = 0; p < passes; ++p) {
    for (size_t i = blockIdx.x * (size_t)PNT + threadIdx.x; i < n4; i += 4 * stride) {
      float4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) v[u] = (i + u * stride < n4) ? __ldcg(src + i + u * stride) : make_float4(0, 0, 0, 0);
#pragma unroll
      for (int u = 0; u < 4; ++u) { acc.x += v[u].x; acc.y += v[u].y; acc.z += v[u].z; acc.w += v[u].w; }
    }
  }
  sink[blockIdx.x * PNT + threadIdx.x] = acc.x + acc.y + acc.z + acc.w;
}

constexpr int FNT = 256;

// The selection round without its work: push h floats into slot [buf][rank]
// of every CTA, barrier, merge the C slots + block reduction, warp 0 pushes a
// short list, barrier, merge the lists.
__global__ void __launch_bounds__(FNT) select_floor_kernel(int h, int rounds, float* __restrict__ sink) {
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank(), C = (int)cluster.num_blocks();
  extern __shared__ float fs[];
  float* slot1 = fs;                       // [2][C][h]
  float* slot2 = slot1 + 2 * C * h;        // [2][C][4]
  float* red = slot2 + 2 * C * 4;          // [FNT / 32]
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float val = (float)tid;
  for (int r = 0; r < rounds; ++r) {
    const int buf = r & 1;
    for (int i = tid; i < h; i += FNT)
      for (int rr = 0; rr < C; ++rr) cluster.map_shared_rank(slot1 + (buf * C + rank) * h, rr)[i] = val + (float)i;
    cluster.sync();
    float acc = 0.f;
    for (int i = tid; i < h; i += FNT)
      for (int c = 0; c < C; ++c) acc += slot1[(buf * C + c) * h + i];
    acc = warp_sum(acc);
    if (lane == 0) red[warp] = acc;
    __syncthreads();
    float s = lane < FNT / 32 ? red[lane] : 0.f;
    s = warp_sum(s);
    if (warp == 0 && lane < C) {
      float* d = cluster.map_shared_rank(slot2 + (buf * C + rank) * 4, lane);
      d[0] = s; d[1] = s + 1.f; d[2] = (float)rank;
    }
    cluster.sync();
    float best = -INFINITY;
    if (warp == 0) {
      const float v = lane < C ? slot2[(buf * C + lane) * 4] : -INFINITY;
      best = warp_max(v);
    }
    __syncthreads();
    val += (warp == 0 ? best : 0.f) * 1e-12f;
    __syncthreads();
  }
  sink[blockIdx.x * FNT + tid] = val;
  cluster.sync();
}

struct Timer {
  cudaEvent_t a = nullptr, b = nullptr;
  Timer() { cudaEventCreate(&a); cudaEventCreate(&b); }
  ~Timer() { if (a) cudaEventDestroy(a); if (b) cudaEventDestroy(b); }
};

}  // namespace

extern "C" {

int bench_probe_smem_gbs(double* gbs) {
  if (!gbs) return (int)cudaErrorInvalidValue;
  const int grid = sm_count() * 2, iters = 4096;
  float* sink = nullptr;
  cudaError_t e = cudaMalloc(&sink, (size_t)grid * PNT * sizeof(float));
  Timer t;
  const size_t smem = SMEM_F4 * sizeof(float4);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(smem_read_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess) {
    smem_read_kernel<<<grid, PNT, smem>>>(iters, sink);  // warm-up
    cudaEventRecord(t.a);
    smem_read_kernel<<<grid, PNT, smem>>>(iters, sink);
    cudaEventRecord(t.b);
    e = cudaEventSynchronize(t.b);
  }
  float ms = 0.f;
  if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, t.a, t.b);
  if (sink) cudaFree(sink);
  if (e != cudaSuccess) return (int)e;
  *gbs = (double)grid * PNT * iters * sizeof(float4) / (ms * 1e-3) / 1e9;
  return 0;
}

int bench_probe_l2_gbs(double* gbs) {
  if (!gbs) return (int)cudaErrorInvalidValue;
  const size_t bytes = (size_t)48 << 20;  // well inside the L2
  const size_t n4 = bytes / sizeof(float4);
  const int grid = sm_count() * 4, passes = 20;
  float4* src = nullptr;
  float* sink = nullptr;
  cudaError_t e = cudaMalloc(&src, bytes);
  if (e == cudaSuccess) e = cudaMalloc(&sink, (size_t)grid * PNT * sizeof(float));
  if (e == cudaSuccess) e = cudaMemset(src, 0, bytes);
  Timer t;
  if (e == cudaSuccess) {
    l2_read_kernel<<<grid, PNT>>>(src, n4, 2, sink);  // warm: the buffer now sits in L2
    cudaEventRecord(t.a);
    l2_read_kernel<<<grid, PNT>>>(src, n4, passes, sink);
    cudaEventRecord(t.b);
    e = cudaEventSynchronize(t.b);
  }
  float ms = 0.f;
  if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, t.a, t.b);
  if (src) cudaFree(src);
  if (sink) cudaFree(sink);
  if (e != cudaSuccess) return (int)e;
  *gbs = (double)bytes * passes / (ms * 1e-3) / 1e9;
  return 0;
}

int bench_probe_select_floor(int cluster_size, int h, int rounds, int episodes, double* us_per_round) {
  if (!us_per_round) return (int)cudaErrorInvalidValue;
  if ((cluster_size != 8 && cluster_size != 16) || h < 128 || h > 1024 || rounds < 1 || episodes < 1 ||
      episodes * cluster_size > 4096)
    return (int)cudaErrorInvalidValue;
  const int C = cluster_size;
  const size_t smem = (size_t)(2 * C * h + 2 * C * 4 + FNT / 32) * sizeof(float);
  float* sink = nullptr;
  cudaError_t e = cudaMalloc(&sink, (size_t)episodes * C * FNT * sizeof(float));
  if (e == cudaSuccess) e = cudaFuncSetAttribute(select_floor_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess && C > 8) e = cudaFuncSetAttribute(select_floor_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(episodes * C, 1, 1);
  cfg.blockDim = dim3(FNT, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  Timer t;
  if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, select_floor_kernel, h, 8, sink);  // warm-up
  if (e == cudaSuccess) {
    cudaEventRecord(t.a);
    e = cudaLaunchKernelEx(&cfg, select_floor_kernel, h, rounds, sink);
    cudaEventRecord(t.b);
  }
  if (e == cudaSuccess) e = cudaEventSynchronize(t.b);
  float ms = 0.f;
  if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, t.a, t.b);
  if (sink) cudaFree(sink);
  if (e != cudaSuccess) return (int)e;
  *us_per_round = (double)ms * 1e3 / rounds;
  return 0;
}

}  // extern "C"
