// tree.h -- structured arguments: validation of a call's argument tree, recipes, and the
// binding of a tree to an op's flat argument tuple (§3.3 of the paper: a recipe binds the
// source arguments to a logical input tree; guards address values by path; the consumed
// leaves are taken out in preorder only after the checks hold).
#pragma once
#include <stdint.h>

#include "trident_scm.h"

namespace trident {

// A validated copy of a recipe, owned by its version.
struct Recipe {
  int32_t nargs = 0;
  int32_t nnodes = 0;
  trident_recipe_node* nodes = nullptr;  // new[]'d copy
  double eps = 0.0, rope_theta = 0.0, scalar = 0.0;
  int32_t op = 0, nslots = 0;
};

// Checks a call's tree: kinds, child ranges (after the parent, inside the array), every
// node reached at most once, size and depth limits, DLTensor fields. Returns a
// trident_status (ERR_INVALID with a message).
int32_t validate_tree(const trident_node* nodes, int32_t nargs, int32_t nnodes);

// Checks a recipe for an op with `nslots` tensor slots and copies it into *out.
int32_t make_recipe(const trident_recipe* r, int32_t op, int32_t nslots, Recipe* out);
void free_recipe(Recipe* r);

// Matches the recipe against a validated tree and, on a match, fills *args (op, slots in
// slot order, eps / theta / scalar). Returns false if the tree's structure or a guarded
// constant differs (this version's miss).
bool bind_tree(const Recipe& r, const trident_node* nodes, int32_t nargs, trident_args* args);

}  // namespace trident
