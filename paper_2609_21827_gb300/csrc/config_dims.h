// config_dims.h -- the kernels' view of a rheo_config, shared by the entry
// points (api.cu defines these) so that every entry point fills the launch
// arguments the same way.
#pragma once

#include "rheo.h"
#include "rheo_kernels.h"

namespace rheo {

// Dimensions of a valid configuration; chunks = the expansion's tiles per row
// (the verification entry points set their own chunk count).
Dims config_dims(const rheo_config& c);
TreePtrs tree_ptrs(const rheo_tree* t);
PrunedPtrs pruned_ptrs(const rheo_pruned* p);

}  // namespace rheo
