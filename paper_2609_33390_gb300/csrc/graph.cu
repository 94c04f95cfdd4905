// A decode tail captured once into a CUDA graph and replayed block after block (the paper's
// CUDA Graph replay of the fused head, App. F). The graph holds every launch of one
// brisk_decode_tail call with the caller's buffers baked in: per block the caller refreshes
// the input buffers in place and launches the graph, which costs one launch on the host
// instead of a dozen. With io->x0 == io->next_anchor the anchor chains on the device from one
// block to the next.
#include <new>

#include "brisk_internal.cuh"

struct brisk_graph {
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
};

extern "C" brisk_status brisk_tail_graph_create(const brisk_dims* dims, const brisk_params* params,
                                                const void* tables, const brisk_tail_io* io,
                                                int32_t select_mode, int32_t verify_mode,
                                                void* workspace, void* stream,
                                                brisk_graph** out) {
  if (!out || !stream) return BRISK_ERR_INVALID_ARG;
  *out = nullptr;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // one direct call first: it checks the arguments, creates the side streams and sets the
  // kernels' attributes, none of which may happen inside a capture
  brisk_status s = brisk_decode_tail(dims, params, tables, io, select_mode, verify_mode, workspace,
                                     nullptr, stream);
  if (s != BRISK_OK) return s;
  if (cudaStreamSynchronize(st) != cudaSuccess) return BRISK_ERR_CUDA;
  brisk_graph* g = new (std::nothrow) brisk_graph();
  if (!g) return BRISK_ERR_CUDA;
  // The side streams belong to the capture from the call's first fork until the end of the
  // capture: hold their lock over the whole of it, so that another thread's call cannot enqueue
  // on them in between (its work would land in this graph, or break the capture).
  std::lock_guard<std::mutex> lock(brisk::side_stream_mutex());
  if (cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
    delete g;
    return BRISK_ERR_CUDA;
  }
  s = brisk::decode_tail_locked(dims, params, tables, io, select_mode, verify_mode, workspace,
                                nullptr, stream);
  const cudaError_t ec = cudaStreamEndCapture(st, &g->graph);
  if (s != BRISK_OK || ec != cudaSuccess ||
      cudaGraphInstantiate(&g->exec, g->graph, 0) != cudaSuccess) {
    if (g->graph) cudaGraphDestroy(g->graph);
    delete g;
    return s != BRISK_OK ? s : BRISK_ERR_CUDA;
  }
  *out = g;
  return BRISK_OK;
}

extern "C" brisk_status brisk_tail_graph_launch(brisk_graph* g, void* stream) {
  if (!g || !g->exec) return BRISK_ERR_INVALID_ARG;
  return cudaGraphLaunch(g->exec, static_cast<cudaStream_t>(stream)) == cudaSuccess ? BRISK_OK
                                                                                   : BRISK_ERR_CUDA;
}

extern "C" void brisk_tail_graph_destroy(brisk_graph* g) {
  if (!g) return;
  if (g->exec) cudaGraphExecDestroy(g->exec);
  if (g->graph) cudaGraphDestroy(g->graph);
  delete g;
}
